// dm_hash.cu -- prompt hashing (Sec. 3.2: two independent hash functions
// over the prompt prefix; App. A.1.1 block-granular keys), and the routing
// kernel that hashes, looks the candidates up on both rings (Sec. 3.2,
// Sec. 3.4, App. A.1.3) and probes their cache indices (App. A.3.2) in one
// pass over the tokens.  The batch layout it reads is made by dm_setup.cu.
//
// Per full block k of a prompt (B tokens t_0..t_{B-1}) under function f:
//   nh^f_k = sum_i ((t_2i + K^f_2i) mod 2^32) * ((t_2i+1 + K^f_2i+1) mod 2^32)  mod 2^64
//   d^f_k  = fmix64(nh^f_k + (k+1) G^f)
//   P^f_b  = sum_{k<=b} d^f_k  mod 2^64
// Because the chain is a plain prefix sum, every 64-block segment of every
// prompt is hashed independently (one warp each); a segment writes its local
// prefix values and its totals, and the carry of the earlier segments is
// added where a key is needed.  f2 only runs over the first K = min(Kf2,
// n_blk) blocks (Kf2 = K_route, or the longest adaptive prefix): segments
// below K write the sum of their f2 digests and, with the adaptive length,
// each block's in-segment f2 prefix value.
#include <atomic>

#include "dm_internal.cuh"

namespace dm {

// ---------------------------------------------------------------------------
// Streaming 16-byte load: read once, not kept in L1; with an L2 evict-first
// policy the token stream does not push the index lines and the previous
// commit's writes out of L2.
__device__ __forceinline__ uint4 ld_stream(const uint4 *p, uint64_t pol) {
    uint4 v;
    asm volatile("ld.global.nc.L1::no_allocate.L2::cache_hint.v4.u32 {%0,%1,%2,%3}, [%4], %5;"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "l"(__cvta_generic_to_global(p)), "l"(pol));
    return v;
}

__device__ __forceinline__ uint64_t evict_first_policy() {
    uint64_t pol;
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol));
    return pol;
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

// Per-lane constants of the segment hash: lane l = g * U + q reduces the
// NH of one block per load instruction; its 4 key words of each function.
template <int U>
struct HashLane {
    static constexpr int GPL = 32 / U;   // blocks per load instruction
    int q, g, bq, src;
    uint32_t k1[4], k2[4];
    uint64_t G1, G2;
    __device__ __forceinline__ HashLane(const DevState &d, int lane) {
        q = lane % U;
        g = lane / U;
        bq = q * GPL + g;                      // block this lane reduces
        src = (lane % GPL) * U + lane / GPL;   // lane holding block `lane` after the reduction
#pragma unroll
        for (int i = 0; i < 4; ++i) { k1[i] = d.K1[4 * q + i]; k2[i] = d.K2[4 * q + i]; }
        G1 = d.G1;
        G2 = d.G2;
    }
};

// One segment of up to 64 blocks (two iterations of 32 blocks): blocks
// b0 .. b0+nb-1 of a prompt whose tokens start at src4 (block b0's first
// token).  Iteration `it` covers 32 blocks (32*U uint4): load j of lane l
// reads uint4 j*32+l of the iteration (fully coalesced), which is quarter
// l%U of block j*(32/U)+l/U.  Both iterations' loads are issued before any
// arithmetic (4 KB in flight per warp at B = 16); load_segment issues them
// and hash_loaded consumes them, so a caller can do other work in between.
template <int U>
__device__ __forceinline__ void load_segment(const HashLane<U> &hl, const uint4 *src4, uint32_t nb, int lane,
                                             uint64_t pol, uint4 (&v)[2][U]) {
    constexpr int GPL = HashLane<U>::GPL;
#pragma unroll
    for (int it = 0; it < 2; ++it)
#pragma unroll
        for (int jj = 0; jj < U; ++jj) {
            const uint32_t blk = it * 32 + jj * GPL + hl.g;
            v[it][jj] = blk < nb ? ld_stream(src4 + uint64_t(it) * 32 * U + jj * 32 + lane, pol)
                                 : make_uint4(0, 0, 0, 0);
        }
}

// After the reduce-scatter lane l holds block (l%U)*(32/U) + l/U; one
// shuffle puts block m on lane m for the scan.  Lane l returns P[it] = the
// local f1 prefix value of block b0 + 32 it + l (0 past the segment) and
// every lane the f1 total; blocks below K also take f2: kF2 sums their
// digests into sum2 (kP2: also each block's in-segment f2 prefix value into
// p2out, indexed from b0).
template <int U, bool kF2, bool kP2>
__device__ __forceinline__ void hash_loaded(const HashLane<U> &hl, const uint4 (&v)[2][U], uint32_t b0, uint32_t nb,
                                            uint32_t K, int lane, uint64_t (&P)[2], uint64_t &tot1, uint64_t &sum2,
                                            uint64_t *p2out) {
    uint64_t carry1 = 0, s2 = 0;   // kP2: s2 is the running f2 prefix (uniform)
#pragma unroll
    for (int it = 0; it < 2; ++it) {
        P[it] = 0;
        if ((uint32_t)it * 32 >= nb) continue;
        const uint32_t nvalid = min(32u, nb - it * 32);
        uint64_t p1[U];
#pragma unroll
        for (int jj = 0; jj < U; ++jj) p1[jj] = nh4(v[it][jj], hl.k1);
        const uint64_t a1 = reduce_scatter<U>(p1, hl.q);
        const uint32_t kb = b0 + it * 32 + hl.bq;   // block index within the prompt
        uint64_t dg1 = (uint32_t)hl.bq < nvalid ? fmix64(a1 + uint64_t(kb + 1) * hl.G1) : 0;
        dg1 = shfl_u64(dg1, hl.src);
        const uint64_t P1 = warp_incl_scan(dg1, lane) + carry1;
        P[it] = (uint32_t)lane < nvalid ? P1 : 0;
        carry1 = shfl_u64(P1, 31);
        if constexpr (kF2) {
            if (b0 + it * 32 < K) {                   // second function, blocks < K
                uint64_t p2[U];
#pragma unroll
                for (int jj = 0; jj < U; ++jj) p2[jj] = nh4(v[it][jj], hl.k2);
                const uint64_t a2 = reduce_scatter<U>(p2, hl.q);
                const uint64_t dg2 =
                    ((uint32_t)hl.bq < nvalid && kb < K) ? fmix64(a2 + uint64_t(kb + 1) * hl.G2) : 0;
                if constexpr (kP2) {
                    const uint64_t P2 = warp_incl_scan(shfl_u64(dg2, hl.src), lane) + s2;
                    if ((uint32_t)lane < nvalid && b0 + it * 32 + lane < K) p2out[it * 32 + lane] = P2;
                    s2 = shfl_u64(P2, 31);
                } else {
                    s2 += dg2;
                }
            }
        }
    }
    if constexpr (kF2 && !kP2) s2 = warp_sum_u64(s2);
    tot1 = carry1;
    sum2 = s2;
}

template <int U, bool kF2, bool kP2>
__device__ __forceinline__ void hash_segment(const HashLane<U> &hl, const uint4 *src4, uint32_t b0, uint32_t nb,
                                             uint32_t K, int lane, uint64_t pol, uint64_t (&P)[2], uint64_t &tot1,
                                             uint64_t &sum2, uint64_t *p2out) {
    uint4 v[2][U];
    load_segment<U>(hl, src4, nb, lane, pol, v);
    hash_loaded<U, kF2, kP2>(hl, v, b0, nb, K, lane, P, tot1, sum2, p2out);
}

// Hashing only (dm_hash_prompts and the allocation-free variant): one warp
// per segment in segment order; writes every block's local prefix value and
// each segment's totals.
template <int U, bool kP2>
__global__ void __launch_bounds__(256, 4) k_hash(DevState d, const uint32_t *__restrict__ tokens) {
    pdl_enter();
    if (has_err(d.err)) return;
    const int lane = threadIdx.x & 31;
    const uint32_t nwarps = (gridDim.x * blockDim.x) >> 5;
    const uint32_t gw = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const uint32_t total_segs = d.info->total_segs;
    const HashLane<U> hl(d, lane);
    const uint64_t pol = evict_first_policy();
    for (uint32_t seg = gw; seg < total_segs; seg += nwarps) {
        const uint32_t r = d.seg_req[seg];
        const uint32_t j = seg - d.r_segoff[r];
        const uint32_t nblk = d.r_nblk[r];
        const uint32_t b0 = j * kSegBlocks;
        const uint32_t nb = min(kSegBlocks, nblk - b0);
        const uint4 *src4 = reinterpret_cast<const uint4 *>(tokens + d.r_tokoff[r] + uint64_t(b0) * d.B);
        const uint64_t bo = d.r_blkoff[r];
        uint64_t P[2], tot1, sum2;
        hash_segment<U, true, kP2>(hl, src4, b0, nb, min(d.Kf2, nblk), lane, pol, P, tot1, sum2,
                                   kP2 ? d.p2local + bo + b0 : nullptr);
        uint64_t *out = d.plocal + bo + b0;
        if ((uint32_t)lane < nb) out[lane] = P[0];
        if ((uint32_t)lane + 32 < nb) out[lane + 32] = P[1];
        if (lane == 0) {
            d.seg_total[seg] = tot1;
            d.seg_total2[seg] = sum2;
        }
    }
}

// Grids of the hashing kernels, per device (SM counts may differ).
namespace {
constexpr int kGridDevices = 64;
std::atomic<int> g_grid[kGridDevices][2];

template <typename K>
int grid_for_device(int which, K kernel) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kGridDevices) return full_grid(kernel, 256);
    int g = g_grid[dev][which].load(std::memory_order_relaxed);
    if (!g) {
        g = full_grid(kernel, 256);
        g_grid[dev][which].store(g, std::memory_order_relaxed);
    }
    return g;
}
}  // namespace

int hash_grid_size() { return grid_for_device(0, k_hash<4, false>); }

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
// Routing: hashing, ring lookup and probes in one kernel.
//
// Task order.  A hashing task is one 64-block segment of one prompt.  First
// come the routing columns: segment j of every request for j < C, column by
// column, where C covers the longest routing prefix; then the rest of every
// request's head (its segments below H, which hold the cached run in the
// workloads here), request after request; then every remaining segment.
//
// Warp roles.  In every CTA kHashWarps warps only hash: grid-stride over the
// tasks, tokens staged through shared memory with cp.async one task ahead
// (the next task's request and layout looked up one task earlier still),
// prefix values and totals stored, and, for a head segment, a checked record
// published for the other warps (SegPub).  The warp that hashes a request's
// last head segment also puts the request's route task on its CTA's queue.
// The CTA's kProbeWarps warps work off that queue, so the dependent memory
// round trips of routing and probing (App. A.3.2's metadata queries) never
// hold up the token stream.  A route task, once every head segment of its
// request is published, sums their carries, computes the two ring
// positions, searches both rings (Sec. 3.4, App. A.1.3), applies the
// distinct fix (Sec. 3.2), and finds the leading run on both candidates:
//   - It tests the first block of every head segment on both candidates.
//     On c_f let j_f be the first head segment whose first block is missing.
//   - A request touches its keys from its last block down (App. A.3.2's
//     save, in arrival order), so a key's last touch always comes after the
//     last touch of every longer prefix of the same prompt, and an exact LRU
//     evicts the longer prefix first: the keys resident on an instance are
//     closed under prefixes (barring a 64-bit key collision between two
//     different prefixes).  So every block before segment j_f - 1 is
//     resident on c_f and the first miss is block 64 j_f or lies in segment
//     j_f - 1, which the route task probes (keys from the segment's stored
//     prefix values when they check against its record, else hashed again
//     from the tokens).  When every head segment's first block is resident
//     the run may go on past the head: it hashes on from there.
// A route task whose head is not published yet goes back on the queue;
// after kRetries tries it moves to a list that the kernel's last CTA to
// finish works off, when everything is published.  Nothing waits on a warp
// of another CTA.  The segment carries of the whole batch, which the commit
// needs, and the route outputs are produced by the choice kernel's launch.

// Request holding task x of a part: the largest r < n with off[r] <= x
// (off: exclusive offsets of that part, nondecreasing, off[0] = 0).  The
// whole warp narrows the range 32 ways per round trip (two for n <= 1024).
__device__ __forceinline__ uint32_t find_req(const uint32_t *off, uint32_t n, uint32_t x, int lane) {
    uint32_t lo = 0, len = n;   // the request lies in [lo, lo + len); off[lo] <= x
    while (len > 1) {
        const uint32_t step = (len + 31) / 32;
        const bool le = (uint32_t)lane * step < len && __ldg(off + lo + lane * step) <= x;
        const uint32_t k = 31 - __clz(__ballot_sync(0xffffffffu, le));   // lane 0 always holds
        lo += k * step;
        len = min(step, len - k * step);
    }
    return lo;
}

// Loads through L2 (data written by other warps during this kernel).
__device__ __forceinline__ void ld_cg2(const void *p, uint64_t &a, uint64_t &b) {
    asm volatile("ld.global.cg.v2.u64 {%0, %1}, [%2];" : "=l"(a), "=l"(b) : "l"(__cvta_generic_to_global(p)));
}
__device__ __forceinline__ void st_v2(void *p, uint64_t a, uint64_t b) {
    asm volatile("st.global.v2.u64 [%0], {%1, %2};" ::"l"(__cvta_generic_to_global(p)), "l"(a), "l"(b) : "memory");
}

__device__ __forceinline__ bool seg_pub_read(const SegPub *p, uint64_t E, uint64_t &t1, uint64_t &t2, uint64_t &pf,
                                             uint64_t &pk, uint64_t &px) {
    uint64_t c;
    ld_cg2(&p->t1, t1, t2);
    ld_cg2(&p->pf, pf, pk);
    ld_cg2(&p->px, px, c);
    return c == (t1 ^ t2 ^ pf ^ pk ^ px ^ E);
}

__device__ __forceinline__ void seg_pub_write(SegPub *p, uint64_t E, uint64_t t1, uint64_t t2, uint64_t pf,
                                              uint64_t pk, uint64_t px) {
    st_v2(&p->t1, t1, t2);
    st_v2(&p->pf, pf, pk);
    st_v2(&p->px, px, t1 ^ t2 ^ pf ^ pk ^ px ^ E);
}

// Both candidates' index buffers and log fronts (as of the batch's start).
struct RouteView {
    const Slot *t1, *t2;
    uint64_t f1, f2;
};

constexpr uint32_t kNoMiss = 0xFFFFFFFFu;
constexpr int kHashWarps = 7, kProbeWarps = 1;   // warp roles of a routing CTA
constexpr int kMinBlocks = 2;                    // resident CTAs per SM the registers are sized for
constexpr uint32_t kQCap = 512;                  // entries of a CTA's task queue
constexpr uint32_t kRetries = 1024;              // tries of a task before it goes to the last CTA

// First miss among blocks base + 32 k + lane (k < 2, one segment) below
// `end` on the candidates flagged (kNoMiss if none).  Whole warp.
__device__ __forceinline__ void probe_segment(const uint64_t (&key)[2], uint32_t base, uint32_t end, bool do1,
                                              bool do2, const RouteView &rv, uint64_t mask, uint32_t *err,
                                              uint64_t lim, int lane, uint32_t &m1, uint32_t &m2) {
    uint64_t home[2];
    Slot s1[2], s2[2];
#pragma unroll
    for (int k = 0; k < 2; ++k) {
        const uint32_t b = base + 32 * k + lane;
        home[k] = group_home(group_anchor(key[k], lane), b, mask);
        const bool inb = b < end;
        s1[k] = (inb && do1) ? load_slot(rv.t1 + home[k]) : Slot{0, 0};
        s2[k] = (inb && do2) ? load_slot(rv.t2 + home[k]) : Slot{0, 0};
    }
    m1 = kNoMiss;
    m2 = kNoMiss;
#pragma unroll
    for (int k = 0; k < 2; ++k) {
        const uint32_t b = base + 32 * k + lane;
        const bool inb = b < end;
        if (do1) {
            const bool miss = inb && !resident_at(rv.t1, mask, key[k], home[k], rv.f1, s1[k], err, lim);
            const uint32_t bal = __ballot_sync(0xffffffffu, miss);
            if (bal && m1 == kNoMiss) m1 = base + 32 * k + __ffs(bal) - 1;
        }
        if (do2) {
            const bool miss = inb && !resident_at(rv.t2, mask, key[k], home[k], rv.f2, s2[k], err, lim);
            const uint32_t bal = __ballot_sync(0xffffffffu, miss);
            if (bal && m2 == kNoMiss) m2 = base + 32 * k + __ffs(bal) - 1;
        }
    }
}

// Cache keys of head segment s of request r (nb blocks, f1 carry `carry`
// into it): lane l gets blocks 64 s + l and 64 s + 32 + l.  The prefix
// values come from plocal when what is visible there checks against the
// segment's record (px), else the segment is hashed here from the tokens.
// Whole warp; not inlined.
template <int U>
__device__ __noinline__ void head_seg_keys(const DevState &d, const uint32_t *tokens, uint64_t pol, uint32_t r,
                                           uint32_t s, uint32_t nb, uint64_t carry, uint64_t px, int lane,
                                           uint64_t *key) {
    const uint32_t b0 = s * kSegBlocks;
    const uint64_t *pl = d.plocal + d.r_blkoff[r] + b0;
    uint64_t P0 = (uint32_t)lane < nb ? __ldcg(pl + lane) : 0;
    uint64_t P1 = (uint32_t)lane + 32 < nb ? __ldcg(pl + lane + 32) : 0;
    uint64_t x = P0 ^ P1;
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) x ^= shfl_xor_u64(x, o);
    if (x != px) {   // some value not visible yet
        const HashLane<U> hl(d, lane);
        const uint4 *src = reinterpret_cast<const uint4 *>(tokens + d.r_tokoff[r] + uint64_t(b0) * d.B);
        uint64_t P[2], tot, s2u;
        hash_segment<U, false, false>(hl, src, b0, nb, 0, lane, pol, P, tot, s2u, nullptr);
        P0 = P[0];
        P1 = P[1];
    }
    key[0] = cache_key(P0 + carry, d.Sc);
    key[1] = cache_key(P1 + carry, d.Sc);
}

// The run past the head, on the candidates whose first miss is still
// kNoMiss (every head block resident there): hashes the prompt on from
// segment j0 (f1 only, from carry `carry`) and probes segment by segment
// until each run ends.  Updates m1 and m2 on every lane (kNoMiss: the whole
// prompt is resident).  Whole warp; not inlined (rare: a cached run longer
// than the head).
template <int U>
__device__ __noinline__ void run_on(const DevState &d, const uint32_t *tokens, uint64_t pol, uint32_t r,
                                    uint32_t nblk, uint32_t j0, uint64_t carry, const RouteView &rv, int lane,
                                    uint32_t &m1, uint32_t &m2) {
    const HashLane<U> hl(d, lane);
    const uint4 *tok4 = reinterpret_cast<const uint4 *>(tokens + d.r_tokoff[r]);
    const uint32_t nseg = (nblk + kSegBlocks - 1) / kSegBlocks;
    const uint64_t mask = d.S - 1;
    for (uint32_t j = j0; j < nseg && (m1 == kNoMiss || m2 == kNoMiss); ++j) {
        const uint32_t c0 = j * kSegBlocks, cn = min(kSegBlocks, nblk - c0);
        uint64_t P[2], tot, s2u;
        hash_segment<U, false, false>(hl, tok4 + uint64_t(c0) * d.B / 4, c0, cn, 0, lane, pol, P, tot, s2u,
                                      nullptr);
        const uint64_t key[2] = {cache_key(P[0] + carry, d.Sc), cache_key(P[1] + carry, d.Sc)};
        uint32_t e1, e2;
        probe_segment(key, c0, c0 + cn, m1 == kNoMiss, m2 == kNoMiss, rv, mask, d.err, d.loop_limit, lane, e1,
                      e2);
        if (m1 == kNoMiss) m1 = e1;
        if (m2 == kNoMiss) m2 = e2;
        carry += tot;
    }
}

// The route task of request r.  Returns false, changing nothing, when a head
// segment of r is not published yet.  Whole warp; not inlined.
template <int U, bool kAdapt>
__device__ __noinline__ bool route_task(const DevState &d, const uint32_t *tokens, uint64_t E, uint64_t pol,
                                        uint32_t r, int lane) {
    const uint32_t nblk = d.r_nblk[r], s0 = d.r_segoff[r];
    const uint32_t nseg = (nblk + kSegBlocks - 1) / kSegBlocks, hs = min(nseg, d.H);
    uint64_t t1 = 0, t2 = 0, pf = 0, pk = 0, px = 0;
    const bool ok = (uint32_t)lane >= hs || seg_pub_read(d.seg_pub + s0 + lane, E, t1, t2, pf, pk, px);
    if (!__all_sync(0xffffffffu, ok)) return false;
    const uint64_t inc1 = warp_incl_scan(t1, lane);
    const uint64_t carry = inc1 - t1;   // lane s: f1 carry into head segment s
    uint64_t pos1, pos2;
    uint32_t K;
    if constexpr (kAdapt) {
        __threadfence();   // the head's prefix values were fenced before their records
        adaptive_positions(d, r, nblk, d.r_blkoff[r], lane, carry, warp_incl_scan(t2, lane) - t2, pos1, pos2, K);
    } else {
        K = min(d.Kroute, nblk);
        const uint32_t sK = (K - 1) / kSegBlocks;
        pos1 = fmix64((shfl_u64(carry, sK) + shfl_u64(pk, sK)) ^ d.Sr1);
        pos2 = fmix64(warp_sum_u64((uint32_t)lane <= sK ? t2 : 0) ^ d.Sr2);
    }
    uint32_t lb1, lb2;
    ring_search2(d, pos1, pos2, lane, lb1, lb2);
    DM_CHECK(lb1 < d.R && lb2 < d.R, d.err);
    const uint32_t a = d.ring[0].owner[lb1];
    const uint32_t raw2 = d.ring[1].owner[lb2];
    const uint32_t b = raw2 != a ? raw2 : d.next_live[a];
    DM_CHECK(a < d.M && b < d.M && a != b, d.err);
    RouteView rv;
    rv.t1 = d.table[a];
    rv.t2 = d.table[b];
    rv.f1 = d.log_front[a];   // resident: record at or after the front (as of the batch's start)
    rv.f2 = d.log_front[b];
    const uint64_t mask = d.S - 1;
    // first block of every head segment on both candidates (lane s: segment s)
    bool miss1 = true, miss2 = true;
    if ((uint32_t)lane < hs) {
        const uint64_t key = cache_key(carry + pf, d.Sc);
        const uint64_t home = group_home(key, 0, mask);   // a segment's first block anchors its own group
        miss1 = !resident_at(rv.t1, mask, key, home, rv.f1, load_slot(rv.t1 + home), d.err, d.loop_limit);
        miss2 = !resident_at(rv.t2, mask, key, home, rv.f2, load_slot(rv.t2 + home), d.err, d.loop_limit);
    }
    // j_f: the first head segment whose first block is missing on c_f (hs:
    // none; lanes >= hs count as missing)
    const uint32_t j1 = __ffs(__ballot_sync(0xffffffffu, miss1)) - 1;
    const uint32_t j2 = __ffs(__ballot_sync(0xffffffffu, miss2)) - 1;
    // the run on c_f ends in segment j_f - 1 or at block 64 j_f (when j_f <
    // hs); probe that segment, once for both candidates when they agree
    uint32_t m1 = j1 == 0 ? 0 : kNoMiss, m2 = j2 == 0 ? 0 : kNoMiss;
#pragma unroll 1
    for (int f = 0; f < 2; ++f) {
        const uint32_t jf = f ? j2 : j1;
        if (jf == 0 || (f == 1 && j2 == j1)) continue;
        const uint32_t s = jf - 1, c0 = s * kSegBlocks, cn = min(kSegBlocks, nblk - c0);
        uint64_t key[2];
        head_seg_keys<U>(d, tokens, pol, r, s, cn, shfl_u64(carry, s), shfl_u64(px, s), lane, key);
        const bool do1 = j1 == jf, do2 = j2 == jf;
        uint32_t e1, e2;
        probe_segment(key, c0, c0 + cn, do1, do2, rv, mask, d.err, d.loop_limit, lane, e1, e2);
        if (do1) m1 = e1 != kNoMiss ? e1 : (j1 < hs ? j1 * kSegBlocks : kNoMiss);
        if (do2) m2 = e2 != kNoMiss ? e2 : (j2 < hs ? j2 * kSegBlocks : kNoMiss);
    }
    // every head block resident on a candidate: its run may go on past the head
    if ((m1 == kNoMiss || m2 == kNoMiss) && hs < nseg)
        run_on<U>(d, tokens, pol, r, nblk, hs, shfl_u64(inc1, hs - 1), rv, lane, m1, m2);
    if (lane == 0) {
        d.r_K[r] = K;
        d.r_c1[r] = a;
        d.r_c2[r] = b;
        d.r_m1[r] = m1;
        d.r_m2[r] = m2;
    }
    return true;
}

// Token staging: a hashing warp streams its tasks' segments through a ring
// of shared-memory stages, kStages - 1 segments ahead of the one it hashes:
// lane 0 issues one bulk copy per segment (cp.async.bulk, completed on the
// stage's mbarrier).  A stage holds the segment's tokens as they lie in
// memory, so lane l reads the same 16-byte pieces as load_segment
// (conflict-free); blocks past the segment are not copied and the hash
// masks them out.
template <int U>
struct HP {
    static constexpr int kWarps = kHashWarps + kProbeWarps;
    static constexpr int kThreads = 32 * kWarps;
    static constexpr uint32_t kStage = 64 * U;   // uint4 per stage: one segment
    static constexpr int kStages = U <= 4 ? 3 : (U == 8 ? 2 : 1);
    static constexpr size_t kSmem = size_t(kHashWarps) * kStages * kStage * sizeof(uint4);
};

__device__ __forceinline__ uint32_t smem_addr(const void *p) { return (uint32_t)__cvta_generic_to_shared(p); }

__device__ __forceinline__ void mbar_init(uint64_t *bar) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(smem_addr(bar)) : "memory");
}

// Lane 0: copy `bytes` (a multiple of 16; both addresses 16-byte aligned)
// from global memory into a stage; the stage's mbarrier completes its
// current phase when they have landed.
__device__ __forceinline__ void bulk_to_stage(uint4 *stage, const uint4 *src, uint32_t bytes, uint64_t *bar,
                                              uint64_t pol) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_addr(bar)), "r"(bytes)
                 : "memory");
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1], %2, [%3], %4;" ::"r"(
            smem_addr(stage)),
        "l"(__cvta_generic_to_global(src)), "r"(bytes), "r"(smem_addr(bar)), "l"(pol)
        : "memory");
}

// Wait (every lane) until the mbarrier's phase with parity `par` completes;
// false after `lim` polls.
__device__ __forceinline__ bool mbar_wait(uint64_t *bar, uint32_t par, uint64_t lim) {
    for (uint64_t k = 0; k < lim; ++k) {
        uint32_t ok;
        asm volatile(
            "{ .reg .pred p; mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2; selp.u32 %0, 1, 0, p; }"
            : "=r"(ok)
            : "r"(smem_addr(bar)), "r"(par)
            : "memory");
        if (ok) return true;
    }
    return false;
}

template <int U>
__device__ __forceinline__ void read_stage(const uint4 *stage, int lane, uint4 (&v)[2][U]) {
#pragma unroll
    for (int it = 0; it < 2; ++it)
#pragma unroll
        for (int jj = 0; jj < U; ++jj) v[it][jj] = stage[(it * U + jj) * 32 + lane];
}

// A CTA's task queue in shared memory: a bounded many-producer,
// many-consumer ring in which every slot carries a sequence number (slot
// k is free for the producer at position p when its number is p, holds
// that producer's entry when it is p + 1, and is free again for position
// p + kQCap once consumed), so neither side ever reads a half-written
// entry.  An entry is a route task: r | (tries + 1) << 32, never 0 (what an
// empty queue returns).
struct CtaQueue {
    uint64_t buf[kQCap];
    uint32_t seq[kQCap];
    uint32_t head, tail;
    uint32_t hash_done;   // hashing warps out of tasks
    uint32_t busy;        // warps inside a route task
};

__device__ __forceinline__ uint64_t qentry(uint32_t r, uint32_t tries) {
    return uint64_t(r) | uint64_t(tries + 1) << 32;   // never 0
}

// Push one entry (one thread); a full queue sends it to the last CTA's list.
__device__ __forceinline__ void q_push(CtaQueue &q, const DevState &d, uint64_t e) {
    uint32_t pos = *(volatile uint32_t *)&q.tail;
    for (uint32_t k = 0; k < (1u << 20); ++k) {
        const uint32_t sq = *(volatile uint32_t *)&q.seq[pos % kQCap];
        const int32_t dif = (int32_t)(sq - pos);
        if (dif == 0) {
            const uint32_t got = atomicCAS(&q.tail, pos, pos + 1);
            if (got == pos) {
                *(volatile uint64_t *)&q.buf[pos % kQCap] = e;
                __threadfence_block();
                *(volatile uint32_t *)&q.seq[pos % kQCap] = pos + 1;
                return;
            }
            pos = got;
        } else if (dif < 0) {
            break;   // full
        } else {
            pos = *(volatile uint32_t *)&q.tail;
        }
    }
    d.fix_list[atomicAdd(&d.info->fix_n, 1u)] = e;
}

// Pop one entry (one thread); 0 when the queue is empty.  A popped entry
// counts its warp busy until the warp is done with it.
__device__ __forceinline__ uint64_t q_pop(CtaQueue &q) {
    uint32_t pos = *(volatile uint32_t *)&q.head;
    for (uint32_t k = 0; k < (1u << 20); ++k) {
        const uint32_t sq = *(volatile uint32_t *)&q.seq[pos % kQCap];
        const int32_t dif = (int32_t)(sq - (pos + 1));
        if (dif == 0) {
            atomicAdd(&q.busy, 1u);
            const uint32_t got = atomicCAS(&q.head, pos, pos + 1);
            if (got == pos) {
                __threadfence_block();
                const uint64_t e = *(volatile uint64_t *)&q.buf[pos % kQCap];
                __threadfence_block();
                *(volatile uint32_t *)&q.seq[pos % kQCap] = pos + kQCap;
                return e;
            }
            atomicSub(&q.busy, 1u);
            pos = got;
        } else if (dif < 0) {
            return 0;   // empty
        } else {
            pos = *(volatile uint32_t *)&q.head;
        }
    }
    return 0;
}

// Request, segment and layout of one hashing task (j = kNoTask: past the
// warp's last task; nb() = 0: nothing to hash, e.g. a routing column past
// the end of the prompt).
constexpr uint32_t kNoTask = 0xFFFFFFFFu;
struct TaskMeta {
    uint32_t r, j, nblk, segoff;
    uint64_t tokoff, bo;
    __device__ __forceinline__ uint32_t nb() const {
        return j != kNoTask && j * kSegBlocks < nblk ? min(kSegBlocks, nblk - j * kSegBlocks) : 0;
    }
};

// A hashing warp's tasks: in each of the three parts (routing columns, head
// rest, tails) its contiguous share of that part's tasks (the gw-th of nhw
// equal runs), in order.  The request of a task in the second and third
// part is found once per part (find_req) and then followed; a request's
// layout is loaded when the request changes.  Whole warp (uniform).
struct TaskCursor {
    uint32_t part, t, hi;     // current part, next task in it, end of this warp's share
    uint32_t r, rbeg, rend;   // parts 1-2: request of task t and its range in the part (r = kNoTask: not found yet)
    TaskMeta lay;             // layout of request lay.r (lay.r = kNoTask: none)
    uint32_t gw, nhw, n, r0, nr;
    uint32_t lo[3], T[3];     // per part: first task of requests r0 .. r0+nr-1 and their task count
    uint32_t Tall[3];         // per part: tasks of the whole batch

    __device__ __forceinline__ void share() {
        t = lo[part] + uint32_t(uint64_t(T[part]) * gw / nhw);
        hi = lo[part] + uint32_t(uint64_t(T[part]) * (gw + 1) / nhw);
        r = kNoTask;
    }
    // The tasks of requests r0_ .. r1_-1 only (a shard of the batch; all of
    // it when r0_ = 0 and r1_ = n_).
    __device__ __forceinline__ void init(const DevState &d, uint32_t gw_, uint32_t nhw_, uint32_t n_, uint32_t ncol,
                                         uint32_t nhr, uint32_t total, uint32_t r0_, uint32_t r1_) {
        gw = gw_;
        nhw = nhw_;
        n = n_;
        r0 = r0_;
        nr = r1_ - r0_;
        Tall[0] = ncol;
        Tall[1] = nhr;
        Tall[2] = total - ncol - nhr;
        lo[0] = 0;
        T[0] = nr * d.Ccols;
        if (r0_ == 0 && r1_ == n_) {
            lo[1] = lo[2] = 0;
            T[1] = Tall[1];
            T[2] = Tall[2];
        } else {
            lo[1] = __ldg(d.r_hoff + r0_);
            lo[2] = __ldg(d.r_toff + r0_);
            T[1] = (r1_ < n_ ? __ldg(d.r_hoff + r1_) : Tall[1]) - lo[1];
            T[2] = (r1_ < n_ ? __ldg(d.r_toff + r1_) : Tall[2]) - lo[2];
        }
        part = 0;
        lay.r = kNoTask;
        share();
    }
    __device__ __forceinline__ TaskMeta next(const DevState &d, int lane) {
        while (t >= hi && part < 2) {
            ++part;
            share();
        }
        TaskMeta m;
        if (t >= hi) {
            m.r = 0;
            m.j = kNoTask;
            m.nblk = m.segoff = 0;
            m.tokoff = m.bo = 0;
            return m;
        }
        uint32_t rr, j;
        if (part == 0) {   // column-major over the shard's requests
            j = t / nr;
            rr = r0 + (t - j * nr);
        } else {
            const uint32_t *off = part == 1 ? d.r_hoff : d.r_toff;
            if (r == kNoTask) {
                r = find_req(off, n, t, lane);
                rbeg = __ldg(off + r);
                rend = r + 1 < n ? __ldg(off + r + 1) : Tall[part];
            }
            while (t >= rend) {   // ends at the last request, whose range ends at Tall[part] > t
                ++r;
                rbeg = rend;
                rend = r + 1 < n ? __ldg(off + r + 1) : Tall[part];
            }
            rr = r;
            j = (part == 1 ? d.Ccols : d.H) + (t - rbeg);
        }
        ++t;
        if (rr != lay.r) {
            lay.r = rr;
            lay.nblk = d.r_nblk[rr];
            lay.segoff = d.r_segoff[rr];
            lay.tokoff = d.r_tokoff[rr];
            lay.bo = d.r_blkoff[rr];
        }
        m = lay;
        m.j = j;
        return m;
    }
};

template <int U, bool kAdapt>
__global__ void __launch_bounds__(HP<U>::kThreads, kMinBlocks) k_hash_probe(const __grid_constant__ DevState d,
                                                                   const uint32_t *__restrict__ tokens, uint64_t E,
                                                                   uint32_t r0, uint32_t r1) {
    pdl_enter();
    extern __shared__ __align__(16) uint4 s_stage[];
    constexpr int S = HP<U>::kStages;
    __shared__ CtaQueue q;
    __shared__ uint64_t s_bar[kHashWarps * S];   // one mbarrier per stage
    __shared__ uint32_t s_go, s_last;
    if (threadIdx.x == 0) {
        s_go = !has_err(d.err);   // one decision per CTA (the CTA meets barriers below)
        q.head = q.tail = q.hash_done = q.busy = 0;
        for (int i = 0; i < kHashWarps * S; ++i) mbar_init(s_bar + i);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    for (uint32_t i = threadIdx.x; i < kQCap; i += blockDim.x) q.seq[i] = i;
    __syncthreads();
    if (!s_go) return;
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    const uint64_t pol = evict_first_policy();
    if (wid < kHashWarps) {
        // ---- hashing warp ----
        const uint32_t nhw = gridDim.x * kHashWarps;
        const uint32_t gw = blockIdx.x * kHashWarps + wid;
        const uint32_t n = d.info->n, ncol = d.info->col_tasks, nhr = d.info->head_segs;
        const uint32_t total = d.info->tasks;
        const HashLane<U> hl(d, lane);
        uint4 *const stage = s_stage + wid * S * HP<U>::kStage;
        uint64_t *const bar = s_bar + wid * S;
        constexpr uint64_t kWaitLimit = 1ull << 24;   // polls of a stage's mbarrier (seconds)
        uint32_t par = 0, pend = 0;                    // per stage: parity of its next phase; copy issued, not waited
        auto issue = [&](const TaskMeta &m, uint32_t slot) {
            const uint32_t nb = m.nb();
            if (nb) {
                if (lane == 0)
                    bulk_to_stage(stage + slot * HP<U>::kStage,
                                  reinterpret_cast<const uint4 *>(tokens + m.tokoff + uint64_t(m.j) * kSegBlocks * d.B),
                                  nb * d.B * 4, bar + slot, pol);
                pend |= 1u << slot;
            }
        };
        TaskCursor cur_t;
        cur_t.init(d, gw, nhw, n, ncol, nhr, total, r0, r1);
        // m[s]: the warp's k-th task + s; the copies of m[0 .. S-2] are
        // issued, m[S-1] is looked up and issued next
        TaskMeta m[S];
#pragma unroll
        for (int s = 0; s < S; ++s) {
            m[s] = cur_t.next(d, lane);
            if (s + 1 < S) issue(m[s], s);
        }
        for (uint32_t k = 0; m[0].j != kNoTask; ++k) {
            issue(m[S - 1], (k + S - 1) % S);
            const TaskMeta mn = cur_t.next(d, lane);
            const TaskMeta &cur = m[0];
            const uint32_t cnb = cur.nb(), slot = k % S;
            if (cnb) {
                if (!mbar_wait(bar + slot, (par >> slot) & 1, kWaitLimit)) {
                    if (lane == 0) set_err(d.err, DM_ERR_TIMEOUT);
                    break;
                }
                par ^= 1u << slot;
                pend &= ~(1u << slot);
                uint4 v[2][U];
                read_stage<U>(stage + slot * HP<U>::kStage, lane, v);
                // the stage's next bulk copy (async proxy) comes after these reads
                asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
                __syncwarp();
                const uint32_t b0 = cur.j * kSegBlocks, seg = cur.segoff + cur.j;
                DM_CHECK(seg < d.max_segs && cur.bo + b0 + cnb <= d.max_blocks, d.err);
                uint64_t P[2], tot1, sum2;
                hash_loaded<U, true, kAdapt>(hl, v, b0, cnb, min(d.Kf2, cur.nblk), lane, P, tot1, sum2,
                                             kAdapt ? d.p2local + cur.bo + b0 : nullptr);
                uint64_t *out = d.plocal + cur.bo + b0;
                if ((uint32_t)lane < cnb) out[lane] = P[0];
                if ((uint32_t)lane + 32 < cnb) out[lane + 32] = P[1];
                if (lane == 0) {
                    d.seg_total[seg] = tot1;
                    d.seg_total2[seg] = sum2;
                    d.seg_req[seg] = cur.r;
                }
                const uint32_t hs = min((cur.nblk + kSegBlocks - 1) / kSegBlocks, d.H);
                if (cur.j < hs) {
                    // publish the head segment: totals, its first block's and
                    // block K-1's prefix values, and the xor of what it stored
                    // in plocal
                    const uint32_t kk = min(d.Kroute, cur.nblk) - 1 - b0;   // block K-1 in this segment, if any
                    const uint64_t pk = shfl_u64(kk < 32 ? P[0] : P[1], kk & 31);
                    const uint64_t pf = shfl_u64(P[0], 0);
                    uint64_t px = P[0] ^ P[1];
#pragma unroll
                    for (int o = 16; o >= 1; o >>= 1) px ^= shfl_xor_u64(px, o);
                    if constexpr (kAdapt) {
                        __threadfence();   // the route task reads the head's prefix values (plocal, p2local) directly
                        __syncwarp();
                    }
                    if (lane == 0) {
                        seg_pub_write(d.seg_pub + seg, E, tot1, sum2, pf, kk < kSegBlocks ? pk : 0, px);
                        if (cur.j + 1 == hs) q_push(q, d, qentry(cur.r, 0));   // the request's route task
                    }
                }
            }
#pragma unroll
            for (int s = 0; s + 1 < S; ++s) m[s] = m[s + 1];
            m[S - 1] = mn;
        }
        // copies still in flight (only after a timeout): let them land
        for (uint32_t s = 0; s < (uint32_t)S; ++s)
            if ((pend >> s) & 1) mbar_wait(bar + s, (par >> s) & 1, kWaitLimit);
        if (lane == 0) atomicAdd(&q.hash_done, 1u);
    }
    {
        // ---- route tasks: the CTA's queue, worked off by its route warp
        // from the start and by its hashing warps once their segments are
        // done, which matters when a batch has many short prompts (bounded:
        // kIdleLimit idle polls in a row, a few seconds at most, then the
        // call ends with DM_ERR_TIMEOUT) ----
        constexpr uint32_t kIdleLimit = 1u << 22;
        for (uint32_t idle = 0;;) {
            uint64_t e = lane == 0 ? q_pop(q) : 0;
            e = shfl_u64(e, 0);
            if (e == 0) {
                // done once the hashing warps are done, no warp holds a task
                // (it might queue it again) and the queue is empty
                const bool fin = *(volatile uint32_t *)&q.hash_done == kHashWarps &&
                                 *(volatile uint32_t *)&q.busy == 0 &&
                                 *(volatile uint32_t *)&q.head == *(volatile uint32_t *)&q.tail;
                if (__shfl_sync(0xffffffffu, fin, 0)) break;
                if (++idle >= kIdleLimit) {
                    if (lane == 0) set_err(d.err, DM_ERR_TIMEOUT);
                    break;
                }
                __nanosleep(idle < 64 ? 64 : 512);
                continue;
            }
            idle = 0;
            const uint32_t r = (uint32_t)e, tries = (uint32_t)(e >> 32) - 1;
            const bool done = route_task<U, kAdapt>(d, tokens, E, pol, r, lane);
            if (lane == 0) {
                if (!done) {
                    // a head segment hashed elsewhere not published yet: back on the queue
                    if (tries + 1 < kRetries) q_push(q, d, qentry(r, tries + 1));
                    else d.fix_list[atomicAdd(&d.info->fix_n, 1u)] = qentry(r, 0);
                    if (tries > 8) __nanosleep(1000);
                }
                atomicSub(&q.busy, 1u);
            }
            __syncwarp();
        }
    }
    // the last CTA to finish works off the list (every head segment is
    // published by then)
    __syncthreads();
    if (threadIdx.x == 0) {
        __threadfence();
        s_last = atomicAdd(&d.info->cta_done, 1u) + 1 == gridDim.x;
    }
    __syncthreads();
    if (!s_last) return;
    __threadfence();
    const uint32_t nf = *(volatile uint32_t *)&d.info->fix_n;
    const uint32_t nw = blockDim.x >> 5;
    for (uint32_t i = wid; i < nf; i += nw)
        if (!route_task<U, kAdapt>(d, tokens, E, pol, (uint32_t)d.fix_list[i], lane) && lane == 0)
            set_err(d.err, DM_ERR_TIMEOUT);   // cannot happen: everything is published by now
}

// Launch shape of the routing kernel per device and block size: its
// shared-memory stages are set up once, the grid fills every SM.
template <int U, bool kAdapt>
static cudaError_t launch_hash_probe_u(const DevState &d, const dm_batch &b, uint64_t E, uint32_t r0, uint32_t r1,
                                       cudaStream_t st) {
    static std::atomic<int> grids[kGridDevices];
    int dev = 0;
    DM_TRY(cudaGetDevice(&dev));
    if (dev < 0 || dev >= kGridDevices) return cudaErrorInvalidDevice;
    int grid = grids[dev].load(std::memory_order_relaxed);
    if (!grid) {
        DM_TRY(cudaFuncSetAttribute(k_hash_probe<U, kAdapt>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    (int)HP<U>::kSmem));
        int sms = 0, per = 0;
        DM_TRY(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev));
        DM_TRY(cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per, k_hash_probe<U, kAdapt>, HP<U>::kThreads,
                                                             HP<U>::kSmem));
        grid = sms * (per > 0 ? per : 1);
        grids[dev].store(grid, std::memory_order_relaxed);
    }
    DM_TRY(launch_pdl(k_hash_probe<U, kAdapt>, grid, HP<U>::kThreads, HP<U>::kSmem, st, d, b.tokens, E, r0, r1));
    return cudaGetLastError();
}

template <bool kAdapt>
static cudaError_t launch_hash_probe_t(const DevState &d, const dm_batch &b, uint64_t E, uint32_t r0, uint32_t r1,
                                       cudaStream_t st) {
    switch (d.B) {
        case 4: return launch_hash_probe_u<1, kAdapt>(d, b, E, r0, r1, st);
        case 8: return launch_hash_probe_u<2, kAdapt>(d, b, E, r0, r1, st);
        case 16: return launch_hash_probe_u<4, kAdapt>(d, b, E, r0, r1, st);
        case 32: return launch_hash_probe_u<8, kAdapt>(d, b, E, r0, r1, st);
        case 64: return launch_hash_probe_u<16, kAdapt>(d, b, E, r0, r1, st);
        default: return cudaErrorInvalidValue;
    }
}

cudaError_t launch_hash_probe(const DevState &d, const dm_batch &b, uint64_t E, uint32_t r0, uint32_t r1,
                              cudaStream_t st) {
    if (b.n == 0 || r0 >= r1) return cudaSuccess;
    return d.ad_step ? launch_hash_probe_t<true>(d, b, E, r0, r1, st) : launch_hash_probe_t<false>(d, b, E, r0, r1, st);
}

// Carries of every segment of the batch and the route outputs (the
// cluster-wide rules' probes need the carries before their choice kernel;
// the pair rules' choice kernels do this in their own launch).
__global__ void k_carries(DevState d, dm_route_out o, uint32_t n) {
    pdl_enter();
    if (has_err(d.err)) return;
    carries_role(d, o, n, blockIdx.x, gridDim.x);
}

cudaError_t launch_carries(const DevState &d, const dm_route_out &o, uint32_t n, cudaStream_t st) {
    if (n == 0) return cudaSuccess;
    DM_TRY(launch_pdl(k_carries, (n + 7) / 8, 256, 0, st, d, o, n));
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// Sharded routing: what the routing kernel produced for requests r0 .. r1-1
// (the local prefix values of their blocks, their segments' f1 totals and
// owners, and per request the hash length, both candidates and both first
// misses), packed into one buffer in that order (8-byte values first, then
// 4-byte ones) or unpacked from it.  Every replica lays the batch out the
// same way, so the ranges line up.
__device__ __forceinline__ void shard_span(const DevState &d, uint32_t r0, uint32_t r1, uint64_t &b0, uint64_t &nb,
                                           uint64_t &s0, uint64_t &ns) {
    const uint32_t n = d.info->n;
    b0 = d.r_blkoff[r0];
    nb = (r1 < n ? d.r_blkoff[r1] : d.info->total_blocks) - b0;
    s0 = d.r_segoff[r0];
    ns = (r1 < n ? d.r_segoff[r1] : d.info->total_segs) - s0;
}

template <bool kExport>
__global__ void k_shard_copy(DevState d, uint32_t r0, uint32_t r1, uint8_t *buf, uint64_t cap, uint64_t *bytes) {
    pdl_enter();
    if (has_err(d.err)) return;
    uint64_t b0, nb, s0, ns;
    shard_span(d, r0, r1, b0, nb, s0, ns);
    const uint64_t nr = r1 - r0;
    const uint64_t need = 8 * (nb + ns) + 4 * (ns + 5 * nr);
    if (kExport && bytes && blockIdx.x == 0 && threadIdx.x == 0) *bytes = need;
    if (need > cap) {
        if (blockIdx.x == 0 && threadIdx.x == 0) set_err(d.err, DM_ERR_CAPACITY);
        return;
    }
    uint64_t *p64 = reinterpret_cast<uint64_t *>(buf);
    uint32_t *p32 = reinterpret_cast<uint32_t *>(buf + 8 * (nb + ns));
    uint32_t *const rq[5] = {d.r_K, d.r_c1, d.r_c2, d.r_m1, d.r_m2};
    const uint64_t total = nb + ns + ns + 5 * nr;
    for (uint64_t i = uint64_t(blockIdx.x) * blockDim.x + threadIdx.x; i < total;
         i += uint64_t(gridDim.x) * blockDim.x) {
        if (i < nb) {
            if (kExport) p64[i] = d.plocal[b0 + i];
            else d.plocal[b0 + i] = p64[i];
        } else if (i < nb + ns) {
            const uint64_t k = i - nb;
            if (kExport) p64[i] = d.seg_total[s0 + k];
            else d.seg_total[s0 + k] = p64[i];
        } else if (i < nb + 2 * ns) {
            const uint64_t k = i - nb - ns;
            if (kExport) p32[k] = d.seg_req[s0 + k];
            else d.seg_req[s0 + k] = p32[k];
        } else {
            const uint64_t k = i - nb - 2 * ns, a = k / nr, r = r0 + k % nr;
            if (kExport) p32[ns + k] = rq[a][r];
            else rq[a][r] = p32[ns + k];
        }
    }
}

cudaError_t launch_shard_copy(const DevState &d, bool exp, uint32_t r0, uint32_t r1, uint8_t *buf, uint64_t cap,
                              uint64_t *bytes, cudaStream_t st) {
    if (r0 >= r1) return cudaSuccess;
    const int grid = 2 * hash_grid_size();
    if (exp) DM_TRY(launch_pdl(k_shard_copy<true>, grid, 256, 0, st, d, r0, r1, buf, cap, bytes));
    else DM_TRY(launch_pdl(k_shard_copy<false>, grid, 256, 0, st, d, r0, r1, buf, cap, bytes));
    return cudaGetLastError();
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
