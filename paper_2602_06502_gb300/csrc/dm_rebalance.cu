// dm_rebalance.cu -- hotspot-aware request rebalancing (Sec. 3.3, Eq.
// "rebalance": B_r^(i->j) = TTFT_{r,i} - TTFT_{r,j}; App. A.1.2).
//
// Hotspots (hot_den * N * W_i > hot_num * sum W over live instances) are
// visited in descending W.  For hotspot i the CTA gathers, in parallel, every
// queued request that has not started, was not moved in this call and could
// still pass the move test, with
// TTFT_{r,i} = work queued up to and including r and TTFT_{r,j} = W_j +
// cost * (L - h_{r,j}) for its other candidate j (h_{r,j} stored at routing,
// or with DM_REBALANCE_FRESH_HITS probed now from the request's keys); sorts
// them by (benefit desc, sequence asc); then one thread walks the list,
// moving r to j while i
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

// DM_REBALANCE_FRESH_HITS: the leading run (blocks) of a queued request's
// keys, held at ring positions koff .. koff+nblk-1 of `ring` (KQ entries),
// that is resident on instance j now (its index and log front at the call;
// App. A.3.2's metadata query).  The resident keys are closed under prefixes
// (touches run from a prompt's last block down into an exact LRU), so the
// first block of every 64-block segment is tested, 32 segments per round,
// and then the one segment that holds the run's end.  Whole warp.
static __device__ __noinline__ uint32_t ring_leading_run(const DevState &d, const uint64_t *ring, uint64_t koff,
                                                  uint32_t nblk, uint32_t j, int lane) {
    const Slot *t = d.table[j];
    const uint64_t front = d.log_front[j], mask = d.S - 1, km = d.KQ - 1;
    const uint32_t nseg = (nblk + kSegBlocks - 1) / kSegBlocks;
    uint32_t js = nseg;   // first segment whose first block is missing (nseg: none)
    for (uint32_t s0 = 0; s0 < nseg; s0 += 32) {
        const uint32_t sg = s0 + lane;
        bool miss = false;
        if (sg < nseg) {
            const uint64_t key = ring[(koff + uint64_t(sg) * kSegBlocks) & km];
            const uint64_t home = group_home(key, 0, mask);   // a segment's first block anchors its own group
            miss = !resident_at(t, mask, key, home, front, load_slot(t + home), d.err, d.loop_limit);
        }
        const uint32_t bal = __ballot_sync(0xffffffffu, miss);
        if (bal) {
            js = s0 + __ffs(bal) - 1;
            break;
        }
    }
    if (js == 0) return 0;
    // the run ends in segment js - 1, or at block 64 js
    const uint32_t c0 = (js - 1) * kSegBlocks, cn = min(kSegBlocks, nblk - c0);
    uint32_t first = 0xFFFFFFFFu;
#pragma unroll
    for (int k = 0; k < 2; ++k) {
        const uint32_t b = 32 * k + lane;
        const uint64_t key = b < cn ? ring[(koff + c0 + b) & km] : 0;
        const uint64_t home = group_home(group_anchor(key, lane), c0 + b, mask);
        const bool miss = b < cn && !resident_at(t, mask, key, home, front, load_slot(t + home), d.err, d.loop_limit);
        const uint32_t bal = __ballot_sync(0xffffffffu, miss);
        if (bal && first == 0xFFFFFFFFu) first = c0 + 32 * k + __ffs(bal) - 1;
    }
    if (first != 0xFFFFFFFFu) return first;
    return js < nseg ? js * kSegBlocks : nblk;
}

constexpr uint32_t kRbStage = 1024;   // candidates staged per sequential pass

// Sequential-pass staging of one chunk of sorted candidates.
struct RbChunk {
    uint64_t seq[kRbStage], work[kRbStage], ttft_i[kRbStage], new_work[kRbStage];
    uint32_t pos[kRbStage], L[kRbStage], c1[kRbStage], c2[kRbStage], h1[kRbStage], h2[kRbStage];
    uint32_t j[kRbStage];
    // moves decided in this chunk: candidate index and target slot, and
    // (DM_REBALANCE_FRESH_HITS) the ring position of its keys on the target
    uint32_t mv_k[kRbStage], mv_slot[kRbStage];
    uint64_t mv_koff[kRbStage];
};

// Dynamic shared memory layout: per instance W (u64), queue tails (u32),
// hot list (u32), state (u8, padded); then the chunk staging; then the sort
// arrays (key u64, seq u64, ttft u64, pos u32) of up to `sort_cap` candidates.
__host__ __device__ inline size_t rb_inst_bytes(uint32_t M) { return (size_t(M) * 17 + 15) / 16 * 16; }
__host__ __device__ inline size_t rb_sort_bytes(uint32_t cap) { return size_t(cap) * 28; }

// Bitonic sort of P (power of two) candidates by (key asc, seq asc) with
// their payloads; the arrays are shared or global memory of this CTA.
__device__ void bitonic_sort(uint64_t *key, uint64_t *seq, uint64_t *tt, uint32_t *pos, uint32_t P) {
    for (uint32_t k = 2; k <= P; k <<= 1) {
        for (uint32_t jj = k >> 1; jj > 0; jj >>= 1) {
            for (uint32_t x = threadIdx.x; x < P; x += blockDim.x) {
                const uint32_t y = x ^ jj;
                if (y > x) {
                    const bool asc = (x & k) == 0;
                    const uint64_t kx = key[x], ky = key[y];
                    const uint64_t sx = seq[x], sy = seq[y];
                    const bool gt = kx > ky || (kx == ky && sx > sy);
                    if (gt == asc) {
                        key[x] = ky; key[y] = kx;
                        seq[x] = sy; seq[y] = sx;
                        const uint64_t t = tt[x]; tt[x] = tt[y]; tt[y] = t;
                        const uint32_t q = pos[x]; pos[x] = pos[y]; pos[y] = q;
                    }
                }
            }
            __syncthreads();
        }
    }
}

// Single CTA of 1024 threads.
__global__ void __launch_bounds__(1024) k_rebalance(DevState d, uint32_t n, uint64_t seq0, uint32_t call,
                                                    dm_migration *out, uint32_t cap, uint32_t *n_out,
                                                    uint32_t sort_cap) {
    pdl_enter();
    extern __shared__ __align__(16) unsigned char smem[];
    __shared__ uint32_t s_w[33];
    __shared__ uint64_t s_u[33];
    __shared__ uint64_t s_sumW;
    __shared__ uint32_t s_nhot, s_cnt, s_nmv, s_stop;
    if (has_err(d.err)) return;
    const uint32_t M = d.M;
    uint64_t *W = reinterpret_cast<uint64_t *>(smem);
    uint32_t *tails = reinterpret_cast<uint32_t *>(W + M);
    uint32_t *hotl = tails + M;
    uint8_t *st = reinterpret_cast<uint8_t *>(hotl + M);
    RbChunk &Ch = *reinterpret_cast<RbChunk *>(smem + rb_inst_bytes(M));
    unsigned char *sort_base = smem + rb_inst_bytes(M) + sizeof(RbChunk);
    uint64_t *sk = reinterpret_cast<uint64_t *>(sort_base);
    uint64_t *ss = sk + sort_cap;
    uint64_t *stt = ss + sort_cap;
    uint32_t *sp = reinterpret_cast<uint32_t *>(stt + sort_cap);

    uint64_t myW = 0;
    uint32_t myN = 0;
    for (uint32_t i = threadIdx.x; i < M; i += blockDim.x) {
        W[i] = d.W[i];
        tails[i] = d.q_tail[i];
        st[i] = d.inst_state[i];
        if (st[i] == 1) { myW += W[i]; ++myN; }
    }
    const uint64_t sumW0 = block_sum_u64(myW, s_u);
    const uint32_t N = (uint32_t)block_sum_u64(myN, s_u);
    // hot list (ids in ascending order), then ranks by (W desc, id asc);
    // none when the double-overload trigger did not fire
    const bool slo_target = (d.rb_flags & DM_REBALANCE_SLO_TARGET) != 0;
    const bool fresh = (d.rb_flags & DM_REBALANCE_FRESH_HITS) != 0 && d.KQ != 0;
    const bool armed = !(d.rb_flags & DM_REBALANCE_DOUBLE_OVERLOAD) || d.info->both_over;
    uint32_t nhot = 0;
    for (uint32_t base = 0; base < M; base += blockDim.x) {
        const uint32_t i = base + threadIdx.x;
        const bool h = armed && i < M && st[i] == 1 &&
                       (slo_target ? W[i] > d.slo : hot(W[i], sumW0, N, d.hot_num, d.hot_den));
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
        QEntry *qi = d.q + uint64_t(i) * d.Q;
        const uint32_t head = d.q_head[i], tail = tails[i];
        // 1) gather the candidates of hotspot i (parallel over its queue)
        uint64_t ahead = 0;
        uint32_t ncand = 0;
        for (uint32_t p0 = head; p0 != tail;) {
            const uint32_t p = p0 + threadIdx.x;
            const bool valid = (uint32_t)(p - head) < (uint32_t)(tail - head);
            QEntry e{};
            if (valid) e = qi[p & (d.Q - 1)];
            uint64_t tot_rem;
            const uint64_t ex = block_excl_u64(valid ? e.remaining : 0, s_u, &tot_rem);
            const uint64_t ttft_i = ahead + ex + (valid ? e.remaining : 0);
            bool elig = valid && e.moved != kTomb && e.moved != call && e.remaining == e.work;
            const uint32_t jj = e.c1 == i ? e.c2 : e.c1;
            uint32_t hj = jj == e.c1 ? e.h1 : e.h2;   // the hit stored at routing
            if (fresh) {
                // probe the other candidate's index now, a warp per entry in
                // turn; the pending batch's own entries keep their stored
                // hit (no commit since their routing: the same probe)
                const bool need = elig && st[jj] == 1 && !(e.seq >= seq0 && e.seq < seq0 + n);
                const int lane = threadIdx.x & 31;
                for (uint32_t m = __ballot_sync(0xffffffffu, need); m; m &= m - 1) {
                    const int src = __ffs(m) - 1;
                    const uint64_t ko = __shfl_sync(0xffffffffu, e.koff, src);
                    const uint32_t nb = __shfl_sync(0xffffffffu, e.L, src) / d.B;
                    const uint32_t tj = __shfl_sync(0xffffffffu, jj, src);
                    // its keys lie in the live part of the ring (written by an earlier commit)
                    DM_CHECK(ko >= d.kr_head[i] && ko + nb <= d.kr_tail[i], d.err);
                    const uint32_t run = ring_leading_run(d, d.kring + uint64_t(i) * d.KQ, ko, nb, tj, lane);
                    if (lane == src) hj = run * d.B;
                }
                if (elig) d.rb_hq[p & (d.Q - 1)] = hj;
            }
            uint64_t key = 0;
            if (elig) {
                const uint32_t j = jj;
                const uint64_t ttft_j = W[j] + cost * (e.L - hj);
                const int64_t B = (int64_t)(ttft_i - ttft_j);
                key = ~(uint64_t(B) ^ 0x8000000000000000ull);   // ascending = benefit descending
                // While hotspot i is walked, W_j only grows (earlier hotspots
                // are done; i's moves add to their targets), so a request
                // that fails the move test now fails it at its turn too.
                // Dropping it changes no move and no stop decision.
                if (!(B > 0 && ttft_j < d.slo)) elig = false;
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
            p0 += min((uint32_t)blockDim.x, (uint32_t)(tail - p0));
        }
        __syncthreads();   // the candidates written in the last pass, before any thread reads them
        if (ncand > d.rb_cap) {
            if (threadIdx.x == 0) set_err(d.err, DM_ERR_CAPACITY);
            return;
        }
        if (ncand == 0) continue;
        // 2) sort by (benefit desc, sequence asc), in shared memory when it fits
        uint32_t P = 1;
        while (P < ncand) P <<= 1;
        if (P <= sort_cap) {
            for (uint32_t c = threadIdx.x; c < P; c += blockDim.x) {
                const bool v = c < ncand;
                sk[c] = v ? d.rb_key[c] : ~0ull;
                ss[c] = v ? d.rb_seq[c] : ~0ull;
                stt[c] = v ? d.rb_ttft[c] : 0;
                sp[c] = v ? d.rb_pos[c] : 0;
            }
            __syncthreads();
            bitonic_sort(sk, ss, stt, sp, P);
            for (uint32_t c = threadIdx.x; c < ncand; c += blockDim.x) {
                d.rb_ttft[c] = stt[c];
                d.rb_pos[c] = sp[c];
            }
        } else {
            for (uint32_t c = ncand + threadIdx.x; c < P; c += blockDim.x) {
                d.rb_key[c] = ~0ull;
                d.rb_seq[c] = ~0ull;
            }
            __syncthreads();
            bitonic_sort(d.rb_key, d.rb_seq, d.rb_ttft, d.rb_pos, P);
        }
        __syncthreads();
        // 3) walk the sorted candidates chunk by chunk: stage, decide (one
        //    thread, shared memory only), apply the moves in parallel
        if (threadIdx.x == 0) s_stop = 0;
        __syncthreads();
        for (uint32_t c0 = 0; c0 < ncand && !s_stop; c0 += kRbStage) {
            const uint32_t m = min(kRbStage, ncand - c0);
            for (uint32_t k = threadIdx.x; k < m; k += blockDim.x) {
                const uint32_t p = d.rb_pos[c0 + k];
                const QEntry e = qi[p & (d.Q - 1)];
                const uint32_t j = e.c1 == i ? e.c2 : e.c1;
                const uint32_t hj = fresh ? d.rb_hq[p & (d.Q - 1)] : (j == e.c1 ? e.h1 : e.h2);
                Ch.seq[k] = e.seq;
                Ch.work[k] = e.work;
                Ch.ttft_i[k] = d.rb_ttft[c0 + k];
                Ch.new_work[k] = cost * (e.L - hj);
                Ch.pos[k] = p;
                Ch.L[k] = e.L;
                Ch.c1[k] = e.c1;
                Ch.c2[k] = e.c2;
                Ch.h1[k] = e.h1;
                Ch.h2[k] = e.h2;
                Ch.j[k] = j;
            }
            __syncthreads();
            if (threadIdx.x == 0) {
                uint64_t sumW = s_sumW;
                uint32_t nmv = 0, stop = 0;
                for (uint32_t k = 0; k < m; ++k) {
                    if (slo_target ? !(W[i] > d.slo) : !hot(W[i], sumW, N, d.hot_num, d.hot_den)) {
                        stop = 1;
                        break;
                    }
                    const uint32_t j = Ch.j[k];
                    if (st[j] != 1) continue;
                    const uint64_t nw = Ch.new_work[k];
                    const uint64_t ttft_j = W[j] + nw;
                    if (!(Ch.ttft_i[k] > ttft_j && ttft_j < d.slo)) continue;
                    const uint32_t slot = tails[j];
                    if (slot - d.q_head[j] >= d.Q) { set_err(d.err, DM_ERR_CAPACITY); stop = 1; break; }
                    if (fresh) {   // its keys move to the target's ring
                        const uint64_t kt = d.kr_tail[j], nb = Ch.L[k] / d.B;
                        if (kt + nb - d.kr_head[j] > d.KQ) { set_err(d.err, DM_ERR_CAPACITY); stop = 1; break; }
                        d.kr_tail[j] = kt + nb;
                        Ch.mv_koff[nmv] = kt;
                    }
                    tails[j] = slot + 1;
                    W[i] -= Ch.work[k];
                    sumW -= Ch.work[k];
                    W[j] += nw;
                    sumW += nw;
                    Ch.mv_k[nmv] = k;
                    Ch.mv_slot[nmv] = slot;
                    ++nmv;
                }
                s_sumW = sumW;
                s_nmv = nmv;
                s_stop = stop;
            }
            __syncthreads();
            const uint32_t cnt0 = s_cnt;
            for (uint32_t t = threadIdx.x; t < s_nmv; t += blockDim.x) {
                const uint32_t k = Ch.mv_k[t];
                const uint32_t j = Ch.j[k];
                QEntry *src = qi + (Ch.pos[k] & (d.Q - 1));
                src->moved = kTomb;
                src->work = 0;
                src->remaining = 0;
                QEntry e;
                e.seq = Ch.seq[k];
                e.work = e.remaining = Ch.new_work[k];
                e.L = Ch.L[k];
                e.c1 = Ch.c1[k];
                e.c2 = Ch.c2[k];
                e.h1 = Ch.h1[k];
                e.h2 = Ch.h2[k];
                e.moved = call;
                e.arrival = src->arrival;   // TTFT still counts from the original arrival
                e.koff = fresh ? Ch.mv_koff[t] : 0;
                d.q[uint64_t(j) * d.Q + (Ch.mv_slot[t] & (d.Q - 1))] = e;
                if (e.seq >= seq0 && e.seq < seq0 + n) {
                    d.r_final[e.seq - seq0] = j;
                    d.info->final_dirty = 1;
                    if (fresh) d.r_koff[e.seq - seq0] = e.koff;   // the commit writes its keys there
                }
                if (cnt0 + t < cap) out[cnt0 + t] = dm_migration{e.seq, i, j};
            }
            __syncthreads();
            if (fresh) {   // an earlier batch's moved request: its keys follow it
                for (uint32_t t = 0; t < s_nmv; ++t) {
                    const uint32_t k = Ch.mv_k[t];
                    if (Ch.seq[k] >= seq0 && Ch.seq[k] < seq0 + n) continue;
                    const uint64_t from = qi[Ch.pos[k] & (d.Q - 1)].koff, to = Ch.mv_koff[t];
                    const uint64_t *sr = d.kring + uint64_t(i) * d.KQ;
                    uint64_t *dr = d.kring + uint64_t(Ch.j[k]) * d.KQ;
                    const uint32_t nb = Ch.L[k] / d.B;
                    for (uint32_t b = threadIdx.x; b < nb; b += blockDim.x)
                        dr[(to + b) & (d.KQ - 1)] = sr[(from + b) & (d.KQ - 1)];
                }
                __syncthreads();
            }
            if (threadIdx.x == 0) s_cnt = cnt0 + s_nmv;
            __syncthreads();
        }
    }
    __syncthreads();
    for (uint32_t i = threadIdx.x; i < M; i += blockDim.x) {
        d.W[i] = W[i];
        d.q_tail[i] = tails[i];
    }
    if (threadIdx.x == 0) *n_out = s_cnt;
}

cudaError_t launch_rebalance(const DevState &d, uint32_t n, uint64_t seq0, uint32_t call,
                             dm_migration *out, uint32_t cap, uint32_t *n_out, cudaStream_t st) {
    // shared memory: per-instance arrays, chunk staging, then as many sort
    // entries (power of two) as the 227 KB budget allows
    const size_t budget = 227 * 1024 - 2048;
    const size_t fixed = rb_inst_bytes(d.M) + sizeof(RbChunk);
    uint32_t sort_cap = 0;
    if (fixed + rb_sort_bytes(256) <= budget) {
        sort_cap = 256;
        while (sort_cap < 8192 && fixed + rb_sort_bytes(sort_cap * 2) <= budget) sort_cap *= 2;
    }
    const size_t smem = fixed + rb_sort_bytes(sort_cap);
    static size_t configured = 0;
    if (smem > configured) {
        cudaError_t e = cudaFuncSetAttribute(k_rebalance, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             (int)smem);
        if (e != cudaSuccess) return e;
        configured = smem;
    }
    DM_TRY(launch_pdl(k_rebalance, 1, 1024, smem, st, d, n, seq0, call, out, cap, n_out, sort_cap));
    return cudaGetLastError();
}

}  // namespace dm
