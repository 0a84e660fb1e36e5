// dm_rebalance.cu -- hotspot-aware request rebalancing (Sec. 3.3, Eq.
// "rebalance": B_r^(i->j) = TTFT_{r,i} - TTFT_{r,j}; App. A.1.2).
//
// Hotspots (hot_den * N * W_i > hot_num * sum W over live instances) are
// visited in descending W.  For hotspot i the CTA gathers, in parallel, every
// queued request that has not started and was not moved in this call, with
// TTFT_{r,i} = work queued up to and including r and TTFT_{r,j} = W_j +
// cost * (L - h_{r,j}) for its other candidate j; sorts them by (benefit
// desc, sequence asc); then one thread walks the list, moving r to j while i
// is still hot, the benefit (re-evaluated with the current W_j) is positive
// and TTFT_{r,j} < SLO.  Moved requests leave a tombstone (zero work) in the
// source queue and are appended to the target queue.
#include "dm_internal.cuh"

namespace dm {

__device__ __forceinline__ bool hot(uint64_t Wi, uint64_t sumW, uint32_t N, uint32_t num, uint32_t den) {
    // den * N * Wi > num * sumW in 128-bit arithmetic
    const uint64_t a = uint64_t(den) * N;
    const uint64_t lo1 = a * Wi, hi1 = __umul64hi(a, Wi);
    const uint64_t lo2 = uint64_t(num) * sumW, hi2 = __umul64hi(uint64_t(num), sumW);
    return hi1 > hi2 || (hi1 == hi2 && lo1 > lo2);
}

__device__ __forceinline__ uint32_t rank_in_block(bool f, uint32_t *s_w, uint32_t &total) {
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    const uint32_t b = __ballot_sync(0xffffffffu, f);
    if (lane == 0) s_w[wid] = __popc(b);
    __syncthreads();
    if (wid == 0) {
        const uint32_t v = lane < (int)(blockDim.x >> 5) ? s_w[lane] : 0;
        uint32_t inc = v;
        for (int dd = 1; dd < 32; dd <<= 1) {
            const uint32_t u = __shfl_up_sync(0xffffffffu, inc, dd);
            if (lane >= dd) inc += u;
        }
        s_w[lane] = inc - v;
        if (lane == 31) s_w[32] = inc;
    }
    __syncthreads();
    const uint32_t r = s_w[wid] + __popc(b & ((1u << lane) - 1));
    total = s_w[32];
    __syncthreads();
    return r;
}

__device__ __forceinline__ uint64_t block_sum_u64(uint64_t v, uint64_t *s) {
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
#pragma unroll
    for (int dd = 16; dd >= 1; dd >>= 1) v += __shfl_xor_sync(0xffffffffu, v, dd);
    if (lane == 0) s[wid] = v;
    __syncthreads();
    uint64_t t = 0;
    for (int w = 0; w < (int)(blockDim.x >> 5); ++w) t += s[w];
    __syncthreads();
    return t;
}

// Exclusive block scan of u64 values; returns exclusive prefix, total in *tot.
__device__ __forceinline__ uint64_t block_excl_u64(uint64_t v, uint64_t *s, uint64_t *tot) {
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    uint64_t inc = warp_incl_scan(v, lane);
    if (lane == 31) s[wid] = inc;
    __syncthreads();
    if (wid == 0) {
        const uint64_t x = lane < (int)(blockDim.x >> 5) ? s[lane] : 0;
        const uint64_t y = warp_incl_scan(x, lane);
        s[lane] = y - x;
        if (lane == 31) s[32] = y;
    }
    __syncthreads();
    const uint64_t r = s[wid] + inc - v;
    *tot = s[32];
    __syncthreads();
    return r;
}

// Single CTA of 1024 threads; dynamic smem: W[M] u64, hot list u32[M].
__global__ void __launch_bounds__(1024) k_rebalance(DevState d, uint32_t n, uint64_t seq0, uint32_t call,
                                                    dm_migration *out, uint32_t cap, uint32_t *n_out) {
    extern __shared__ __align__(16) unsigned char smem[];
    __shared__ uint32_t s_w[33];
    __shared__ uint64_t s_u[33];
    __shared__ uint64_t s_sumW;
    __shared__ uint32_t s_nhot, s_cnt;
    if (has_err(d.err)) return;
    uint64_t *W = reinterpret_cast<uint64_t *>(smem);
    uint32_t *hotl = reinterpret_cast<uint32_t *>(W + d.M);
    uint64_t myW = 0;
    uint32_t myN = 0;
    for (uint32_t i = threadIdx.x; i < d.M; i += blockDim.x) {
        W[i] = d.W[i];
        if (d.inst_state[i] == 1) { myW += W[i]; ++myN; }
    }
    const uint64_t sumW0 = block_sum_u64(myW, s_u);
    const uint32_t N = (uint32_t)block_sum_u64(myN, s_u);
    // hot list (ids in ascending order), then ranks by (W desc, id asc)
    uint32_t nhot = 0;
    for (uint32_t base = 0; base < d.M; base += blockDim.x) {
        const uint32_t i = base + threadIdx.x;
        const bool h = i < d.M && d.inst_state[i] == 1 && hot(W[i], sumW0, N, d.hot_num, d.hot_den);
        uint32_t tot;
        const uint32_t rk = rank_in_block(h, s_w, tot);
        if (h) d.rb_pos[nhot + rk] = i;   // scratch: unsorted hot ids
        nhot += tot;
    }
    __syncthreads();
    for (uint32_t a = threadIdx.x; a < nhot; a += blockDim.x) {
        const uint32_t x = d.rb_pos[a];
        uint32_t rk = 0;
        for (uint32_t b = 0; b < nhot; ++b) {
            const uint32_t y = d.rb_pos[b];
            rk += (W[y] > W[x]) || (W[y] == W[x] && y < x);
        }
        hotl[rk] = x;
    }
    if (threadIdx.x == 0) { s_sumW = sumW0; s_cnt = 0; s_nhot = nhot; }
    __syncthreads();
    const uint64_t cost = d.cost;
    for (uint32_t hi = 0; hi < s_nhot; ++hi) {
        const uint32_t i = hotl[hi];
        const QEntry *qi = d.q + uint64_t(i) * d.Q;
        const uint32_t head = d.q_head[i], tail = d.q_tail[i];
        uint64_t ahead = 0;
        uint32_t ncand = 0;
        for (uint32_t p0 = head; p0 != tail && (uint32_t)(p0 - head) < (uint32_t)(tail - head);) {
            const uint32_t p = p0 + threadIdx.x;
            const bool valid = (uint32_t)(p - head) < (uint32_t)(tail - head);
            QEntry e{};
            if (valid) e = qi[p & (d.Q - 1)];
            uint64_t tot_rem;
            const uint64_t ex = block_excl_u64(valid ? e.remaining : 0, s_u, &tot_rem);
            const uint64_t ttft_i = ahead + ex + (valid ? e.remaining : 0);
            const bool elig = valid && e.moved != kTomb && e.moved != call && e.remaining == e.work;
            uint64_t key = 0;
            if (elig) {
                const uint32_t j = e.c1 == i ? e.c2 : e.c1;
                const uint32_t hj = j == e.c1 ? e.h1 : e.h2;
                const uint64_t ttft_j = W[j] + cost * (e.L - hj);
                const int64_t B = (int64_t)(ttft_i - ttft_j);
                key = ~(uint64_t(B) ^ 0x8000000000000000ull);   // ascending = benefit descending
            }
            uint32_t tot;
            const uint32_t rk = rank_in_block(elig, s_w, tot);
            if (elig) {
                const uint32_t c = ncand + rk;
                if (c < d.rb_cap) {
                    d.rb_key[c] = key;
                    d.rb_seq[c] = e.seq;
                    d.rb_ttft[c] = ttft_i;
                    d.rb_pos[c] = p;
                }
            }
            ncand += tot;
            ahead += tot_rem;
            const uint32_t step = min((uint32_t)blockDim.x, (uint32_t)(tail - p0));
            p0 += step;
        }
        if (ncand > d.rb_cap) {
            if (threadIdx.x == 0) set_err(d.err, DM_ERR_CAPACITY);
            return;
        }
        // bitonic sort of the candidates by (key asc, seq asc), padded to a power of two
        uint32_t P = 1;
        while (P < ncand) P <<= 1;
        for (uint32_t c = ncand + threadIdx.x; c < P; c += blockDim.x) {
            d.rb_key[c] = ~0ull;
            d.rb_seq[c] = ~0ull;
        }
        __syncthreads();
        for (uint32_t k = 2; k <= P; k <<= 1) {
            for (uint32_t jj = k >> 1; jj > 0; jj >>= 1) {
                for (uint32_t x = threadIdx.x; x < P; x += blockDim.x) {
                    const uint32_t y = x ^ jj;
                    if (y > x) {
                        const bool asc = (x & k) == 0;
                        const uint64_t kx = d.rb_key[x], ky = d.rb_key[y];
                        const uint64_t sx = d.rb_seq[x], sy = d.rb_seq[y];
                        const bool gt = kx > ky || (kx == ky && sx > sy);
                        if (gt == asc) {
                            d.rb_key[x] = ky; d.rb_key[y] = kx;
                            d.rb_seq[x] = sy; d.rb_seq[y] = sx;
                            const uint64_t tx = d.rb_ttft[x];
                            d.rb_ttft[x] = d.rb_ttft[y]; d.rb_ttft[y] = tx;
                            const uint32_t px = d.rb_pos[x];
                            d.rb_pos[x] = d.rb_pos[y]; d.rb_pos[y] = px;
                        }
                    }
                }
                __syncthreads();
            }
        }
        if (threadIdx.x == 0) {
            uint64_t sumW = s_sumW;
            uint32_t cnt = s_cnt;
            for (uint32_t c = 0; c < ncand; ++c) {
                if (!hot(W[i], sumW, N, d.hot_num, d.hot_den)) break;
                const uint32_t p = d.rb_pos[c];
                QEntry *pe = d.q + uint64_t(i) * d.Q + (p & (d.Q - 1));
                QEntry e = *pe;
                const uint32_t j = e.c1 == i ? e.c2 : e.c1;
                if (d.inst_state[j] != 1) continue;
                const uint32_t hj = j == e.c1 ? e.h1 : e.h2;
                const uint64_t new_work = cost * (e.L - hj);
                const uint64_t ttft_j = W[j] + new_work;
                if (!(d.rb_ttft[c] > ttft_j && ttft_j < d.slo)) continue;
                const uint32_t slot = d.q_tail[j];
                if (slot - d.q_head[j] >= d.Q) { set_err(d.err, DM_ERR_CAPACITY); break; }
                pe->moved = kTomb;
                pe->work = 0;
                pe->remaining = 0;
                W[i] -= e.work;
                sumW -= e.work;
                e.work = e.remaining = new_work;
                e.moved = call;
                d.q[uint64_t(j) * d.Q + (slot & (d.Q - 1))] = e;
                d.q_tail[j] = slot + 1;
                W[j] += new_work;
                sumW += new_work;
                if (e.seq >= seq0 && e.seq < seq0 + n) {
                    d.r_final[e.seq - seq0] = j;
                    d.info->final_dirty = 1;
                }
                if (cnt < cap) out[cnt] = dm_migration{e.seq, i, j};
                ++cnt;
            }
            s_sumW = sumW;
            s_cnt = cnt;
        }
        __syncthreads();
    }
    __syncthreads();
    for (uint32_t i = threadIdx.x; i < d.M; i += blockDim.x) d.W[i] = W[i];
    if (threadIdx.x == 0) *n_out = s_cnt;
}

cudaError_t launch_rebalance(const DevState &d, uint32_t n, uint64_t seq0, uint32_t call,
                             dm_migration *out, uint32_t cap, uint32_t *n_out, cudaStream_t st) {
    const size_t smem = size_t(d.M) * (sizeof(uint64_t) + sizeof(uint32_t));
    static size_t configured = 0;
    if (smem > configured) {
        cudaError_t e = cudaFuncSetAttribute(k_rebalance, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             (int)smem);
        if (e != cudaSuccess) return e;
        configured = smem;
    }
    k_rebalance<<<1, 1024, smem, st>>>(d, n, seq0, call, out, cap, n_out);
    return cudaGetLastError();
}

}  // namespace dm
