// dm_choice.cu -- the SLO-aware choice (Sec. 3.2; App. A.1.1: TTFT(r,i) =
// T_q(r,i) + T_c(r,i)), the rules it is compared with (Sec. 2.2, Sec. 4.3),
// and the serving metrics sampled at choice time (Sec. 2.2 CV; Sec. 4.1).
//
// Queues: instance i owns a ring buffer of Q entries with monotonically
// increasing head/tail counters; W[i] is the sum of remaining work.
//
// Choice between two candidates (DualMap's rule and the pair variants):
// the decision for a request depends on the loads left by every earlier
// request of the batch that shares one of its candidates.  One CTA keeps W
// in shared memory; one warp decides 32 requests at a time in dependency
// rounds (a request waits only for earlier requests of the window sharing
// an instance with it); everything that does not depend on W is precomputed
// in parallel, and queue writes and outputs are emitted in parallel
// afterwards.
//
// Cluster-wide rules: every request depends on every earlier one, so one
// warp decides them one at a time (an argmin over the live instances),
// with the hits on every live instance probed beforehand by k_probe_all.
//
// At the end of the file: routing with d candidates (App. A.8).
#include "dm_internal.cuh"

namespace dm {

// ---------------------------------------------------------------------------
// Block-wide helpers of the single-CTA choice kernels (1024 threads).

__device__ __forceinline__ unsigned __int128 shfl_xor_u128(unsigned __int128 v, int o) {
    const uint64_t lo = shfl_xor_u64((uint64_t)v, o), hi = shfl_xor_u64((uint64_t)(v >> 64), o);
    return ((unsigned __int128)hi << 64) | lo;
}

struct MetricSums {
    uint64_t tokens, hits, sw, est;
};

// Sums each thread's per-request counters and this thread's share of the
// live instances' S1 = sum W, S2 = sum W^2 and count over the block; one
// thread adds the counters to the metrics (fire-and-forget atomics) and
// leaves the sums as the batch's pending CV sample.  Called by all threads.
__device__ void finish_metrics(const DevState &d, uint32_t n, MetricSums ms, unsigned __int128 S1,
                               unsigned __int128 S2, uint32_t cnt) {
    __shared__ unsigned long long s_u[32][5];
    __shared__ unsigned __int128 s_w[32][2];
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    uint64_t v[5] = {ms.tokens, ms.hits, ms.sw, ms.est, cnt};
#pragma unroll
    for (int j = 0; j < 5; ++j) v[j] = warp_sum_u64(v[j]);
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) {
        S1 += shfl_xor_u128(S1, o);
        S2 += shfl_xor_u128(S2, o);
    }
    if (lane == 0) {
#pragma unroll
        for (int j = 0; j < 5; ++j) s_u[wid][j] = v[j];
        s_w[wid][0] = S1;
        s_w[wid][1] = S2;
    }
    __syncthreads();
    if (wid == 0) {
        // lane w takes warp w's partials; one more warp reduction
        const int nw = (blockDim.x + 31) >> 5;
        uint64_t t[5];
#pragma unroll
        for (int j = 0; j < 5; ++j) t[j] = warp_sum_u64(lane < nw ? s_u[lane][j] : 0);
        unsigned __int128 a = lane < nw ? s_w[lane][0] : 0, b = lane < nw ? s_w[lane][1] : 0;
#pragma unroll
        for (int o = 16; o >= 1; o >>= 1) {
            a += shfl_xor_u128(a, o);
            b += shfl_xor_u128(b, o);
        }
        if (lane != 0) return;
        DevMetrics *m = d.metrics;
        atomicAdd(&m->requests, (unsigned long long)n);
        atomicAdd(&m->prompt_tokens, (unsigned long long)t[0]);
        atomicAdd(&m->hit_tokens, (unsigned long long)t[1]);
        atomicAdd(&m->switched, (unsigned long long)t[2]);
        atomicAdd(&m->est_slo_met, (unsigned long long)t[3]);
        m->pend_n = t[4];
        m->pend_s1[0] = (uint64_t)a;
        m->pend_s1[1] = (uint64_t)(a >> 64);
        m->pend_s2[0] = (uint64_t)b;
        m->pend_s2[1] = (uint64_t)(b >> 64);
        m->pend = 1;
    }
}


constexpr uint32_t kChoiceChunk = 1024;

// Single CTA (1024 threads).  Dynamic shared memory: per instance W (u64),
// a packed counter PT = (log records this batch << 32) | queue tail, so one
// 64-bit add per request advances both, and a lane mask used to find
// conflicts inside a window; then the per-chunk request staging.
//
// Each request is staged as (a, b): a = the candidate with more cached
// blocks (c1 on equal hits), u = uncached work on each, and
// thr = SLO - u_a (-1 when u_a alone exceeds the SLO or the hits are equal),
// so the rule of Sec. 3.2 becomes: choose b iff W_b < W_a and W_a > thr
// (ttft_a = W_a + u_a > SLO); the SLO switch fired iff hits differ and
// W_a > thr.  The pair variants use the general form: choose b iff
// W_a > thr and (k_b < k_a or (k_b == k_a and tieb)), with k = W (+ u when
// the rule compares TTFTs) and tieb set where a tie goes to b (= c1).
struct ChoiceStage {
    uint64_t ua[kChoiceChunk], ub[kChoiceChunk];
    int64_t thr[kChoiceChunk];
    uint64_t Wa[kChoiceChunk], Wb[kChoiceChunk], pt[kChoiceChunk];
    uint32_t ab[kChoiceChunk];     // a | b << 14 | (a is c2) << 28 | (hits differ) << 29 | tieb << 30 | addu << 31
    uint32_t nb[kChoiceChunk];
    uint8_t pickb[kChoiceChunk];
};

// W and PT (8 bytes each), the lane masks padded to a multiple of 4 entries
// so that the staging block starts on a 16-byte boundary for any M.
__host__ __device__ inline size_t choice_lanes(uint32_t M) { return (size_t(M) + 3) / 4 * 4; }
size_t choice_smem(uint32_t M) { return size_t(M) * 16 + choice_lanes(M) * 4 + sizeof(ChoiceStage); }

// kPairRules: the general form (the pair variants and global cache
// affinity); false compiles DualMap's rule alone.
template <bool kPairRules>
__global__ void __launch_bounds__(1024) k_choice(DevState d, dm_route_out o, uint32_t n, uint64_t seq0,
                                                 uint64_t t_batch) {
    pdl_enter();
    extern __shared__ __align__(16) unsigned char smem[];
    if (has_err(d.err)) return;
    if (blockIdx.x > 0) {   // beside the choice: the segment carries the commit needs
        carries_role(d, o, n, blockIdx.x - 1, gridDim.x - 1);
        return;
    }
    uint64_t *W = reinterpret_cast<uint64_t *>(smem);
    uint64_t *PT = W + d.M;
    uint32_t *lanes = reinterpret_cast<uint32_t *>(PT + d.M);
    ChoiceStage &S = *reinterpret_cast<ChoiceStage *>(lanes + choice_lanes(d.M));
    uint32_t live_bits = 0;   // bit k: instance threadIdx.x + k * blockDim.x is live (M <= 8 * 1024)
    for (uint32_t i = threadIdx.x, k = 0; i < d.M; i += blockDim.x, ++k) {
        W[i] = d.W[i];
        PT[i] = d.q_tail[i];
        lanes[i] = 0;
        live_bits |= uint32_t(d.inst_state[i] == 1) << k;
    }
    const uint64_t cost = d.cost, slo = d.slo;
    const uint32_t rule = kPairRules ? d.rule : uint32_t(DM_RULE_DUALMAP);
    MetricSums ms{0, 0, 0, 0};
    for (uint32_t base = 0; base < n; base += kChoiceChunk) {
        const uint32_t m = min(kChoiceChunk, n - base);
        __syncthreads();
        for (uint32_t k = threadIdx.x; k < m; k += blockDim.x) {
            const uint32_t r = base + k;
            const uint32_t L = d.r_L[r], nblk = d.r_nblk[r];
            const uint32_t h1 = hit_tokens(d.r_m1[r], nblk, d.B), h2 = hit_tokens(d.r_m2[r], nblk, d.B);
            const uint32_t c1 = d.r_c1[r], c2 = d.r_c2[r];
            // global cache affinity always takes c1: orient it as a, never b
            const bool a2 = rule != DM_RULE_CACHE_AFFINITY && h2 > h1;
            const bool differ = h1 != h2;
            const uint64_t ua = cost * (L - (a2 ? h2 : h1)), ub = cost * (L - (a2 ? h1 : h2));
            constexpr int64_t kNever = INT64_MAX;   // W_a never exceeds it: keep a
            int64_t thr = -1;
            bool tieb = false, addu = false;
            const bool affine = rule == DM_RULE_PAIR_CACHE_AFFINITY ||
                                (rule == DM_RULE_PAIR_PREBLE && 2ull * max(h1, h2) > L);
            if (rule == DM_RULE_DUALMAP) {
                thr = (!differ || ua > slo) ? -1 : (int64_t)min(slo - ua, (uint64_t)kNever);
            } else if (rule == DM_RULE_CACHE_AFFINITY) {
                thr = kNever;
            } else if (affine) {
                thr = differ ? kNever : -1;
            } else {                       // least loaded / min TTFT (and Preble below half)
                tieb = a2;
                addu = rule != DM_RULE_PAIR_LEAST_LOADED;
            }
            S.ua[k] = ua;
            S.ub[k] = ub;
            S.thr[k] = thr;
            S.ab[k] = (a2 ? c2 : c1) | ((a2 ? c1 : c2) << 14) | (uint32_t(a2) << 28) | (uint32_t(differ) << 29) |
                      (uint32_t(tieb) << 30) | (uint32_t(addu) << 31);
            S.nb[k] = nblk;
        }
        __syncthreads();
        if (threadIdx.x < 32) {
            // Warp 0 takes 32 requests at a time.  A lane may decide once
            // every earlier lane sharing one of its candidates has decided;
            // lanes decided in the same round share no instance, so reading
            // W and writing W[choice] then equals arrival order exactly.
            const int lane = threadIdx.x;
            for (uint32_t w0 = 0; w0 < m; w0 += 32) {
                const uint32_t k = w0 + lane;
                const bool valid = k < m;
                const uint32_t ab = valid ? S.ab[k] : 0;
                const uint32_t a = ab & 0x3FFF, b = (ab >> 14) & 0x3FFF;
                if (valid) {
                    atomicOr(&lanes[a], 1u << lane);
                    atomicOr(&lanes[b], 1u << lane);
                }
                __syncwarp();
                const uint32_t conf = valid ? (lanes[a] | lanes[b]) & ((1u << lane) - 1) : 0;
                __syncwarp();
                if (valid) { lanes[a] = 0; lanes[b] = 0; }
                const uint64_t ua = valid ? S.ua[k] : 0, ub = valid ? S.ub[k] : 0;
                const int64_t thr = valid ? S.thr[k] : 0;
                const bool tieb = (ab >> 30) & 1u;
                const uint64_t xa = (ab >> 31) ? ua : 0, xb = (ab >> 31) ? ub : 0;
                const uint64_t inc = valid ? (uint64_t(S.nb[k]) << 32) + 1 : 0;   // PT step of this request
                uint64_t oWa = 0, oWb = 0, oP = 0;   // the lane's decision, stored once the window is done
                bool opb = false;
                uint32_t done = __ballot_sync(0xffffffffu, !valid);
                while (done != 0xffffffffu) {
                    const bool ready = !((done >> lane) & 1u) && (conf & ~done) == 0;
                    if (ready) {
                        const uint64_t Wa = W[a], Wb = W[b], Pa = PT[a], Pb = PT[b];
                        bool pb;
                        if constexpr (kPairRules) {
                            const uint64_t ka = Wa + xa, kb = Wb + xb;
                            pb = (int64_t)Wa > thr && (kb < ka || (kb == ka && tieb));
                        } else {
                            pb = Wb < Wa && (int64_t)Wa > thr;
                        }
                        const uint32_t ch = pb ? b : a;
                        const uint64_t Pold = pb ? Pb : Pa;
                        W[ch] = pb ? Wb + ub : Wa + ua;
                        PT[ch] = Pold + inc;
                        oWa = Wa;
                        oWb = Wb;
                        oP = Pold;
                        opb = pb;
                    }
                    __syncwarp();
                    done |= __ballot_sync(0xffffffffu, ready);
                }
                if (valid) {
                    S.Wa[k] = oWa;
                    S.Wb[k] = oWb;
                    S.pt[k] = oP;
                    S.pickb[k] = opb;
                }
            }
        }
        __syncthreads();
        for (uint32_t k = threadIdx.x; k < m; k += blockDim.x) {
            const uint32_t r = base + k;
            const uint32_t ab = S.ab[k];
            const uint32_t a = ab & 0x3FFF, b = (ab >> 14) & 0x3FFF;
            const bool a_is_c2 = (ab >> 28) & 1, differ = (ab >> 29) & 1;
            const bool pb = S.pickb[k];
            const uint32_t ch = pb ? b : a;
            const uint64_t ta = S.Wa[k] + S.ua[k], tb = S.Wb[k] + S.ub[k];
            o.ttft1[r] = a_is_c2 ? tb : ta;
            o.ttft2[r] = a_is_c2 ? ta : tb;
            const bool sw = differ && (rule == DM_RULE_DUALMAP ? (int64_t)S.Wa[k] > S.thr[k] : pb);
            o.chosen[r] = ch;
            o.switched[r] = sw;
            d.r_final[r] = ch;
            const uint32_t L = d.r_L[r], nbr = d.r_nblk[r];
            const uint32_t h1 = hit_tokens(d.r_m1[r], nbr, d.B), h2 = hit_tokens(d.r_m2[r], nbr, d.B);
            ms.tokens += L;
            ms.hits += (ch == (a_is_c2 ? b : a)) ? h1 : h2;
            ms.sw += sw;
            ms.est += (pb ? tb : ta) <= slo;
            if (ta > slo && tb > slo) d.info->both_over = 1;
            d.r_touchoff[r] = S.pt[k] >> 32;          // offset among this batch's records of ch
            const uint32_t slot = (uint32_t)S.pt[k];
            if (slot - d.q_head[ch] >= d.Q) {
                set_err(d.err, DM_ERR_CAPACITY);
                continue;
            }
            QEntry e;
            e.seq = seq0 + r;
            e.work = e.remaining = pb ? S.ub[k] : S.ua[k];
            e.L = L;
            e.c1 = a_is_c2 ? b : a;
            e.c2 = a_is_c2 ? a : b;
            e.h1 = h1;
            e.h2 = h2;
            e.moved = 0;
            e.arrival = t_batch;
            // its keys' ring position: the instance's ring tail at the batch's
            // start plus this batch's earlier blocks queued there (the same
            // order as its touch records)
            e.koff = d.KQ ? d.kr_tail[ch] + (S.pt[k] >> 32) : 0;
            if (d.KQ) d.r_koff[r] = e.koff;
            DM_CHECK(ch < d.M, d.err);
            d.q[uint64_t(ch) * d.Q + (slot & (d.Q - 1))] = e;
        }
    }
    __syncthreads();
    unsigned __int128 S1 = 0, S2 = 0;
    uint32_t cnt = 0;
    for (uint32_t i = threadIdx.x, k = 0; i < d.M; i += blockDim.x, ++k) {
        d.W[i] = W[i];
        d.q_tail[i] = (uint32_t)PT[i];
        d.log_adv[i] = PT[i] >> 32;
        if (d.KQ) {   // the batch's keys on instance i take its ring's next positions
            const uint64_t nt = d.kr_tail[i] + (PT[i] >> 32);
            if (nt - d.kr_head[i] > d.KQ) set_err(d.err, DM_ERR_CAPACITY);
            d.kr_tail[i] = nt;
        }
        if ((live_bits >> k) & 1u) {
            S1 += W[i];
            S2 += (unsigned __int128)W[i] * W[i];
            ++cnt;
        }
    }
    if (threadIdx.x == 0) d.info->final_dirty = 0;
    finish_metrics(d, n, ms, S1, S2, cnt);
}

// ---------------------------------------------------------------------------
// Cluster-wide rules.

// Hit tokens of every request on every live instance (0 elsewhere), against
// the index as of the start of the batch: one warp per (request, instance)
// pair, grid-stride.  The first step tests 32 blocks (most instances miss
// block 0), later steps 128 (4 independent lookups per lane); a slot that
// holds the key or is empty settles the lookup at its home slot, anything
// else takes the full probe order.
constexpr int kAllBlock = 256;

__global__ void __launch_bounds__(kAllBlock) k_probe_all(DevState d, uint32_t n) {
    pdl_enter();
    if (has_err(d.err)) return;
    const int lane = threadIdx.x & 31;
    const uint64_t nw = uint64_t(gridDim.x) * (kAllBlock / 32);
    const uint64_t total = uint64_t(n) * d.M;
    const uint64_t mask = d.S - 1;
    for (uint64_t p = (uint64_t(blockIdx.x) * kAllBlock + threadIdx.x) / 32; p < total; p += nw) {
        const uint32_t r = (uint32_t)(p / d.M), i = (uint32_t)(p - uint64_t(r) * d.M);
        uint32_t h = 0;
        if (d.inst_state[i] == 1) {
            const uint32_t nblk = d.r_nblk[r], s0 = d.r_segoff[r];
            const uint64_t bo = d.r_blkoff[r];
            const Slot *t = d.table[i];
            const uint64_t front = d.log_front[i];
            for (uint32_t base = 0, step = 1;; base += 32 * step, step = 4) {
                uint64_t key[4], home[4];
                Slot sl[4];
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    const uint32_t b = base + 32 * j + lane;   // windows of 32 keep the groups whole
                    const bool inb = j < (int)step && b < nblk;
                    key[j] = inb ? cache_key(d.plocal[bo + b] + d.seg_carry[s0 + b / kSegBlocks], d.Sc) : 0;
                    home[j] = group_home(group_anchor(key[j], lane), b, mask);
                    if (inb) sl[j] = load_slot(t + home[j]);
                }
                uint32_t miss_at = 0xFFFFFFFFu;
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    const bool res = key[j] != 0 && resident_at(t, mask, key[j], home[j], front, sl[j], d.err, d.loop_limit);
                    const uint32_t m = __ballot_sync(0xffffffffu, !res);
                    if (j < (int)step && m && miss_at == 0xFFFFFFFFu) miss_at = base + 32 * j + __ffs(m) - 1;
                }
                if (miss_at != 0xFFFFFFFFu) {
                    h = miss_at;
                    break;
                }
            }
        }
        if (lane == 0) d.h_all[p] = h * d.B;
    }
}

// k_choice_global: W and PT per instance and the live ids, then, for a
// chunk of `cap` requests, their per-request fields, their decisions and
// their hits on every live instance; cap is what the shared memory holds
// (at most 1024).  The decisions are written out in parallel after each
// chunk's sequential pass, which touches shared memory only.
__host__ __device__ inline size_t global_stage_off(uint32_t M) { return (size_t(M) * 20 + 15) / 16 * 16; }
constexpr uint32_t kGlobalReqBytes = 64;   // per-request fields and decision
constexpr uint32_t kGlobalReqMax = 1024;

__global__ void __launch_bounds__(1024) k_choice_global(DevState d, dm_route_out o, uint32_t n, uint64_t seq0,
                                                        uint64_t t_batch, uint32_t smem_bytes) {
    pdl_enter();
    extern __shared__ __align__(16) unsigned char smem[];
    __shared__ uint32_t s_wcnt[32];
    if (has_err(d.err)) return;
    uint64_t *W = reinterpret_cast<uint64_t *>(smem);
    uint64_t *PT = W + d.M;
    uint32_t *live = reinterpret_cast<uint32_t *>(PT + d.M);
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    // live ids in ascending order
    uint32_t nl = 0;
    for (uint32_t base = 0; base < d.M; base += blockDim.x) {
        const uint32_t i = base + threadIdx.x;
        const bool f = i < d.M && d.inst_state[i] == 1;
        if (i < d.M) {
            W[i] = d.W[i];
            PT[i] = d.q_tail[i];
        }
        const uint32_t bal = __ballot_sync(0xffffffffu, f);
        if (lane == 0) s_wcnt[wid] = __popc(bal);
        __syncthreads();
        uint32_t off = nl;
        for (int w = 0; w < wid; ++w) off += s_wcnt[w];
        if (f) live[off + __popc(bal & ((1u << lane) - 1))] = i;
        uint32_t tot = 0;
        for (int w = 0; w < (int)(blockDim.x >> 5); ++w) tot += s_wcnt[w];
        nl += tot;
        __syncthreads();
    }
    const size_t off = global_stage_off(d.M);
    const uint64_t fit = (smem_bytes - off) / (kGlobalReqBytes + 4ull * max(nl, 1u));
    const uint32_t cap = fit < kGlobalReqMax ? (uint32_t)fit : kGlobalReqMax;
    uint64_t *s_pold = reinterpret_cast<uint64_t *>(smem + off);
    uint64_t *s_t1 = s_pold + cap, *s_t2 = s_t1 + cap, *s_wa = s_t2 + cap;
    uint32_t *s_L = reinterpret_cast<uint32_t *>(s_wa + cap);
    uint32_t *s_nb = s_L + cap, *s_c1 = s_nb + cap, *s_c2 = s_c1 + cap, *s_h1 = s_c2 + cap, *s_h2 = s_h1 + cap;
    uint32_t *s_ch = s_h2 + cap, *s_hch = s_ch + cap, *s_hits = s_hch + cap;
    const uint64_t cost = d.cost, slo = d.slo;
    const uint32_t rule = d.rule;
    MetricSums ms{0, 0, 0, 0};
    for (uint32_t r0 = 0; cap > 0 && r0 < n; r0 += cap) {
        const uint32_t m = min(cap, n - r0);
        __syncthreads();
        for (uint32_t x = threadIdx.x; x < m * nl; x += blockDim.x) {
            const uint32_t rr = x / nl, k = x - rr * nl;
            s_hits[x] = d.h_all[uint64_t(r0 + rr) * d.M + live[k]];
        }
        for (uint32_t rr = threadIdx.x; rr < m; rr += blockDim.x) {
            const uint32_t r = r0 + rr;
            s_L[rr] = d.r_L[r];
            s_nb[rr] = d.r_nblk[r];
            s_c1[rr] = d.r_c1[r];
            s_c2[rr] = d.r_c2[r];
            s_h1[rr] = hit_tokens(d.r_m1[r], s_nb[rr], d.B);
            s_h2[rr] = hit_tokens(d.r_m2[r], s_nb[rr], d.B);
        }
        __syncthreads();
        if (wid == 0) {
            for (uint32_t rr = 0; rr < m; ++rr) {
                const uint32_t L = s_L[rr];
                const uint32_t *hr = s_hits + rr * nl;
                bool affine = false;
                uint32_t hmax = 0;
                if (rule == DM_RULE_PREBLE) {
                    for (uint32_t k = lane; k < nl; k += 32) hmax = max(hmax, hr[k]);
                    hmax = __reduce_max_sync(0xffffffffu, hmax);
                    affine = 2ull * hmax > L;
                }
                // smallest (key, list index): a lane visits its indices in
                // ascending order, so a strict comparison keeps its lowest;
                // across lanes three 32-bit reductions give the exact pair
                uint64_t bk = ~0ull;
                uint32_t bkk = 0xFFFFFFFFu;
                for (uint32_t k = lane; k < nl; k += 32) {
                    const uint32_t h = hr[k];
                    const uint64_t w = W[live[k]];
                    uint64_t key;
                    if (rule == DM_RULE_LEAST_LOADED) key = w;
                    else if (affine) key = h == hmax ? w : ~0ull;
                    else key = w + cost * (L - h);
                    if (key < bk || bkk == 0xFFFFFFFFu) { bk = key; bkk = k; }
                }
                const uint32_t khi = __reduce_min_sync(0xffffffffu, (uint32_t)(bk >> 32));
                const uint32_t klo =
                    __reduce_min_sync(0xffffffffu, (uint32_t)(bk >> 32) == khi ? (uint32_t)bk : 0xFFFFFFFFu);
                const uint32_t kk = __reduce_min_sync(
                    0xffffffffu, bk == ((uint64_t(khi) << 32) | klo) ? bkk : 0xFFFFFFFFu);
                if (lane == 0 && kk >= nl) {   // no live instance (the host requires two)
                    set_err(d.err, DM_ERR_NO_INSTANCES);
                    s_ch[rr] = 0xFFFFFFFFu;
                } else if (lane == 0) {
                    const uint32_t ch = live[kk], h = hr[kk];
                    s_t1[rr] = W[s_c1[rr]] + cost * (L - s_h1[rr]);
                    s_t2[rr] = W[s_c2[rr]] + cost * (L - s_h2[rr]);
                    const uint64_t Pold = PT[ch];
                    const uint64_t wa = W[ch] + cost * (L - h);
                    W[ch] = wa;
                    PT[ch] = Pold + (uint64_t(s_nb[rr]) << 32) + 1;
                    s_ch[rr] = ch;
                    s_hch[rr] = h;
                    s_pold[rr] = Pold;
                    s_wa[rr] = wa;
                }
                __syncwarp();
            }
        }
        __syncthreads();
        for (uint32_t rr = threadIdx.x; rr < m; rr += blockDim.x) {
            const uint32_t r = r0 + rr, ch = s_ch[rr], L = s_L[rr], h = s_hch[rr];
            if (ch == 0xFFFFFFFFu) continue;
            const uint64_t Pold = s_pold[rr];
            o.ttft1[r] = s_t1[rr];
            o.ttft2[r] = s_t2[rr];
            o.chosen[r] = ch;
            o.switched[r] = 0;
            d.r_final[r] = ch;
            d.r_touchoff[r] = Pold >> 32;
            ms.tokens += L;
            ms.hits += h;
            ms.est += s_wa[rr] <= slo;
            if (s_t1[rr] > slo && s_t2[rr] > slo) d.info->both_over = 1;
            const uint32_t slot = (uint32_t)Pold;
            if (slot - d.q_head[ch] >= d.Q) {
                set_err(d.err, DM_ERR_CAPACITY);
                continue;
            }
            QEntry e;
            e.seq = seq0 + r;
            e.work = e.remaining = cost * (L - h);
            e.L = L;
            e.c1 = s_c1[rr];
            e.c2 = s_c2[rr];
            e.h1 = s_h1[rr];
            e.h2 = s_h2[rr];
            e.moved = 0;
            e.arrival = t_batch;
            e.koff = 0;
            DM_CHECK(ch < d.M, d.err);
            d.q[uint64_t(ch) * d.Q + (slot & (d.Q - 1))] = e;
        }
    }
    if (cap == 0 && threadIdx.x == 0) set_err(d.err, DM_ERR_CAPACITY);   // not even one request fits
    __syncthreads();
    unsigned __int128 S1 = 0, S2 = 0;
    uint32_t cnt = 0;
    for (uint32_t i = threadIdx.x; i < d.M; i += blockDim.x) {
        d.W[i] = W[i];
        d.q_tail[i] = (uint32_t)PT[i];
        d.log_adv[i] = PT[i] >> 32;
        if (d.inst_state[i] == 1) {
            S1 += W[i];
            S2 += (unsigned __int128)W[i] * W[i];
            ++cnt;
        }
    }
    if (threadIdx.x == 0) d.info->final_dirty = 0;
    finish_metrics(d, n, ms, S1, S2, cnt);
}

cudaError_t launch_choice(const DevState &d, const dm_route_out &o, uint32_t n, uint64_t seq0, uint64_t t_batch,
                          cudaStream_t st) {
    if (n == 0) return cudaSuccess;
    if (d.rule >= DM_RULE_LEAST_LOADED) {
        // as much shared memory as the device allows, up to what 1024 requests need
        static uint32_t smem_g = 0, smem_M = 0;
        if (smem_M != d.M) {
            int dev = 0, optin = 0;
            cudaFuncAttributes fa{};
            DM_TRY(cudaGetDevice(&dev));
            DM_TRY(cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev));
            DM_TRY(cudaFuncGetAttributes(&fa, k_choice_global));
            const size_t want = global_stage_off(d.M) + size_t(kGlobalReqMax) * (kGlobalReqBytes + 4ull * d.M);
            const size_t room = size_t(optin) - fa.sharedSizeBytes;
            smem_g = (uint32_t)(want < room ? want : room);
            DM_TRY(cudaFuncSetAttribute(k_choice_global, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem_g));
            smem_M = d.M;
        }
        DM_TRY(launch_carries(d, o, n, st));
        DM_TRY(launch_pdl(k_probe_all, full_grid(k_probe_all, kAllBlock), kAllBlock, 0, st, d, n));
        DM_TRY(launch_pdl(k_choice_global, 1, 1024, smem_g, st, d, o, n, seq0, t_batch, smem_g));
        return cudaGetLastError();
    }
    const size_t smem = choice_smem(d.M);
    static size_t configured = 0;
    if (smem > configured) {
        for (auto k : {k_choice<false>, k_choice<true>}) {
            cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
            if (e != cudaSuccess) return e;
        }
        configured = smem;
    }
    // CTA 0 decides; CTAs 1.. sum the batch's segment carries meanwhile (a warp per request)
    const unsigned grid = 1 + (n + 31) / 32 < 1 + 152 ? 1 + (n + 31) / 32 : 1 + 152;
    if (d.rule == DM_RULE_DUALMAP)
        DM_TRY(launch_pdl(k_choice<false>, grid, 1024, smem, st, d, o, n, seq0, t_batch));
    else
        DM_TRY(launch_pdl(k_choice<true>, grid, 1024, smem, st, d, o, n, seq0, t_batch));
    return cudaGetLastError();
}


// ---------------------------------------------------------------------------
// Routing with d candidates instead of two (App. A.8,
// "Optimal Candidate Set Size": the paper weighs d and keeps d = 2; this is
// the d-way version of the path, for that comparison).  After the plain
// hashing kernel (f1 chained prefix values and totals):
//   k_route_d   warp per request: segment carries, the d ring positions
//               (function 1 from the prefix values; functions 2..d hash the
//               first K blocks here), a successor search on each ring, the
//               distinct fix, and the leading run of resident blocks on
//               each candidate;
//   k_choice_d  one CTA: DualMap's SLO-aware rule over d candidates in
//               arrival order (one thread; this path is for experiments,
//               not the benchmark), queue appends, the commit's per-request
//               offsets and the batch's metrics, exactly as k_choice leaves
//               them for d = 2.


// Index (level 0) of the successor of p on ring f.  Whole warp.
__device__ __forceinline__ uint32_t ring_search1(const DevState &d, int f, uint64_t p, int lane) {
    const int top = (int)d.nlev - 1;
    const uint64_t nt = d.lev_n[top];
    const uint64_t vt = (uint64_t)lane < nt ? level_ptr(d, f, top)[lane] : ~0ull;
    int64_t i = (int64_t)__popc(__ballot_sync(0xffffffffu, vt < p)) - 1;
    for (int k = top - 1; k >= 0; --k) {
        const uint64_t nk = d.lev_n[k];
        const uint64_t a = (uint64_t)(i < 0 ? 0 : i) * 32 + lane;
        const uint64_t v = (i >= 0 && a < nk) ? level_ptr(d, f, k)[a] : ~0ull;
        const int c = __popc(__ballot_sync(0xffffffffu, v < p));
        if (i >= 0) i = i * 32 + c - 1;
    }
    return (uint32_t)(i + 1 == (int64_t)d.R ? 0 : i + 1);
}

// NH key word j of function f (0-based).
__device__ __forceinline__ uint32_t nh_key(const DevState &d, uint32_t f, uint32_t j) {
    return f == 0 ? d.K1[j] : f == 1 ? d.K2[j] : d.Kx[(f - 2) * 64 + j];
}

__global__ void k_route_d(DevState d, const uint32_t *tokens, uint32_t n) {
    pdl_enter();
    if (has_err(d.err)) return;
    const int lane = threadIdx.x & 31;
    const uint32_t r = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    if (r >= n) return;
    request_carries(d, r, lane);
    __syncwarp();
    const uint32_t nblk = d.r_nblk[r], s0 = d.r_segoff[r], B = d.B, nd = d.nd;
    const uint64_t bo = d.r_blkoff[r];
    const uint32_t K = min(d.Kroute, nblk);
    const uint32_t *tok = tokens + d.r_tokoff[r];
    uint32_t cand[kMaxD];
    for (uint32_t f = 0; f < nd; ++f) {
        uint64_t P;
        if (f == 0) {
            P = d.plocal[bo + K - 1] + d.seg_carry[s0 + (K - 1) / kSegBlocks];
        } else {   // function f over the first K blocks: a lane per block
            const uint64_t G = f == 1 ? d.G2 : d.Gx[f - 2];
            uint64_t acc = 0;
            for (uint32_t b = lane; b < K; b += 32) {
                uint64_t nh = 0;
                for (uint32_t i = 0; i < B; i += 2)
                    nh += uint64_t(tok[uint64_t(b) * B + i] + nh_key(d, f, i)) *
                          uint64_t(tok[uint64_t(b) * B + i + 1] + nh_key(d, f, i + 1));
                acc += fmix64(nh + uint64_t(b + 1) * G);
            }
            P = warp_sum_u64(acc);
        }
        const uint64_t Sr = f == 0 ? d.Sr1 : f == 1 ? d.Sr2 : d.Srx[f - 2];
        uint32_t x = d.ring[f].owner[ring_search1(d, (int)f, fmix64(P ^ Sr), lane)];
        for (uint32_t k = 0; k < nd; ++k) {   // taken by an earlier ring: the next live id after it
            bool taken = false;
            for (uint32_t g = 0; g < f; ++g) taken |= cand[g] == x;
            if (!taken) break;
            x = d.next_live[x];
        }
        cand[f] = x;
    }
    // leading run of resident blocks on each candidate (index as of the start of the batch)
    const uint64_t mask = d.S - 1;
    for (uint32_t f = 0; f < nd; ++f) {
        const Slot *t = d.table[cand[f]];
        const uint64_t front = d.log_front[cand[f]];
        uint32_t h = nblk;
        for (uint32_t base = 0; base < nblk; base += 32) {
            const uint32_t b = base + lane;
            const bool inb = b < nblk;
            const uint64_t key = inb ? cache_key(d.plocal[bo + b] + d.seg_carry[s0 + b / kSegBlocks], d.Sc) : 0;
            const uint64_t home = group_home(group_anchor(key, lane), b, mask);
            const bool miss = inb && !resident_at(t, mask, key, home, front, load_slot(t + home), d.err, d.loop_limit);
            const uint32_t bal = __ballot_sync(0xffffffffu, miss);
            if (bal) {
                h = base + __ffs(bal) - 1;
                break;
            }
        }
        if (lane == 0) {
            d.rd_cand[uint64_t(r) * nd + f] = cand[f];
            d.rd_hit[uint64_t(r) * nd + f] = h * B;
        }
    }
    if (lane == 0) d.r_K[r] = K;
}

// DualMap's rule over d candidates, in arrival order (one thread), then the
// batch's loads, queue tails, commit offsets and metrics as k_choice leaves
// them.  Dynamic shared memory: W and the packed (records << 32 | queue
// tail) counter of every instance.
__global__ void __launch_bounds__(1024) k_choice_d(DevState d, dm_route_out_d o, uint32_t n, uint64_t seq0,
                                                   uint64_t t_batch) {
    pdl_enter();
    extern __shared__ __align__(16) unsigned char smem[];
    if (has_err(d.err)) return;
    uint64_t *W = reinterpret_cast<uint64_t *>(smem);
    uint64_t *PT = W + d.M;
    uint32_t live_bits = 0;
    for (uint32_t i = threadIdx.x, k = 0; i < d.M; i += blockDim.x, ++k) {
        W[i] = d.W[i];
        PT[i] = d.q_tail[i];
        live_bits |= uint32_t(d.inst_state[i] == 1) << k;
    }
    __syncthreads();
    const uint32_t nd = d.nd;
    const uint64_t cost = d.cost, slo = d.slo;
    uint64_t tokens = 0, hits = 0, sw = 0, est = 0;
    if (threadIdx.x == 0) {
        for (uint32_t r = 0; r < n; ++r) {
            const uint32_t *c = d.rd_cand + uint64_t(r) * nd, *h = d.rd_hit + uint64_t(r) * nd;
            const uint32_t L = d.r_L[r];
            uint32_t hmax = 0, nmax = 0, a = 0;
            for (uint32_t f = 0; f < nd; ++f) hmax = max(hmax, h[f]);
            bool all_over = true, first = true;
            for (uint32_t f = 0; f < nd; ++f) {
                const uint64_t t = W[c[f]] + cost * (L - h[f]);
                o.ttft[uint64_t(r) * nd + f] = t;
                all_over = all_over && t > slo;
                if (h[f] == hmax) {
                    ++nmax;
                    if (first || W[c[f]] < W[c[a]]) a = f;
                    first = false;
                }
            }
            uint32_t pick = a;
            const bool over = nmax < nd && W[c[a]] + cost * (L - h[a]) > slo;
            if (over)
                for (uint32_t f = 0; f < nd; ++f)
                    if (W[c[f]] < W[c[pick]]) pick = f;
            const uint32_t ch = c[pick];
            const uint64_t u = cost * (L - h[pick]);
            o.chosen[r] = ch;
            o.switched[r] = over;
            for (uint32_t f = 0; f < nd; ++f) {
                o.cand[uint64_t(r) * nd + f] = c[f];
                o.hit[uint64_t(r) * nd + f] = h[f];
            }
            if (all_over) d.info->both_over = 1;
            const uint64_t Pold = PT[ch];
            W[ch] += u;
            PT[ch] = Pold + (uint64_t(d.r_nblk[r]) << 32) + 1;
            d.r_final[r] = ch;
            d.r_touchoff[r] = Pold >> 32;   // offset among this batch's records of ch
            tokens += L;
            hits += h[pick];
            sw += over;
            est += W[ch] <= slo;
            const uint32_t slot = (uint32_t)Pold;
            if (slot - d.q_head[ch] >= d.Q) {
                set_err(d.err, DM_ERR_CAPACITY);
                continue;
            }
            QEntry e;
            e.seq = seq0 + r;
            e.work = e.remaining = u;
            e.L = L;
            e.c1 = c[0];
            e.c2 = nd > 1 ? c[1] : c[0];
            e.h1 = h[0];
            e.h2 = nd > 1 ? h[1] : h[0];
            e.moved = 0;
            e.arrival = t_batch;
            e.koff = 0;
            DM_CHECK(ch < d.M, d.err);
            d.q[uint64_t(ch) * d.Q + (slot & (d.Q - 1))] = e;
        }
    }
    __syncthreads();
    unsigned __int128 S1 = 0, S2 = 0;
    uint32_t cnt = 0;
    for (uint32_t i = threadIdx.x, k = 0; i < d.M; i += blockDim.x, ++k) {
        d.W[i] = W[i];
        d.q_tail[i] = (uint32_t)PT[i];
        d.log_adv[i] = PT[i] >> 32;
        if ((live_bits >> k) & 1u) {
            S1 += W[i];
            S2 += (unsigned __int128)W[i] * W[i];
            ++cnt;
        }
    }
    if (threadIdx.x == 0) d.info->final_dirty = 0;
    finish_metrics(d, n, MetricSums{tokens, hits, sw, est}, S1, S2, cnt);
}

cudaError_t launch_route_d(const DevState &d, const dm_batch &b, const dm_route_out_d &o, uint64_t seq0,
                           cudaStream_t st) {
    if (b.n == 0) return cudaSuccess;
    DM_TRY(launch_pdl(k_route_d, (b.n + 7) / 8, 256, 0, st, d, b.tokens, b.n));
    const size_t smem = size_t(d.M) * 16;
    static size_t configured = 0;
    if (smem > configured) {
        DM_TRY(cudaFuncSetAttribute(k_choice_d, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
        configured = smem;
    }
    DM_TRY(launch_pdl(k_choice_d, 1, 1024, smem, st, d, o, b.n, seq0, b.batch_time_us));
    return cudaGetLastError();
}

}  // namespace dm
