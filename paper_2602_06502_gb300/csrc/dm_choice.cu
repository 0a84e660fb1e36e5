// dm_choice.cu -- queue draining and the SLO-aware choice (Sec. 3.2;
// App. A.1.1: TTFT(r,i) = T_q(r,i) + T_c(r,i)).
//
// Queues: instance i owns a ring buffer of Q entries with monotonically
// increasing head/tail counters; W[i] is the sum of remaining work.
//
// Choice: the decision for a request depends on the loads left by every
// earlier request of the batch that shares one of its candidates.  One CTA
// keeps W in shared memory; one warp decides 32 requests at a time in
// dependency rounds (a request waits only for earlier requests of the window
// sharing an instance with it); everything that does not depend on W is
// precomputed in parallel, and queue writes and outputs are emitted in
// parallel afterwards.
#include "dm_internal.cuh"

namespace dm {


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
// W_a > thr.
struct ChoiceStage {
    uint64_t ua[kChoiceChunk], ub[kChoiceChunk];
    int64_t thr[kChoiceChunk];
    uint64_t Wa[kChoiceChunk], Wb[kChoiceChunk], pt[kChoiceChunk];
    uint32_t ab[kChoiceChunk];     // a | b << 14 | (a is c2) << 28 | (hits differ) << 29
    uint32_t nb[kChoiceChunk];
    uint8_t pickb[kChoiceChunk];
};

// W and PT (8 bytes each), the lane masks padded to a multiple of 4 entries
// so that the staging block starts on a 16-byte boundary for any M.
__host__ __device__ inline size_t choice_lanes(uint32_t M) { return (size_t(M) + 3) / 4 * 4; }
size_t choice_smem(uint32_t M) { return size_t(M) * 16 + choice_lanes(M) * 4 + sizeof(ChoiceStage); }

__global__ void __launch_bounds__(1024) k_choice(DevState d, dm_route_out o, uint32_t n, uint64_t seq0) {
    pdl_enter();
    extern __shared__ __align__(16) unsigned char smem[];
    if (has_err(d.err)) return;
    uint64_t *W = reinterpret_cast<uint64_t *>(smem);
    uint64_t *PT = W + d.M;
    uint32_t *lanes = reinterpret_cast<uint32_t *>(PT + d.M);
    ChoiceStage &S = *reinterpret_cast<ChoiceStage *>(lanes + choice_lanes(d.M));
    for (uint32_t i = threadIdx.x; i < d.M; i += blockDim.x) {
        W[i] = d.W[i];
        PT[i] = d.q_tail[i];
        lanes[i] = 0;
    }
    const uint64_t cost = d.cost, slo = d.slo;
    for (uint32_t base = 0; base < n; base += kChoiceChunk) {
        const uint32_t m = min(kChoiceChunk, n - base);
        __syncthreads();
        for (uint32_t k = threadIdx.x; k < m; k += blockDim.x) {
            const uint32_t r = base + k;
            const uint32_t L = d.r_L[r], h1 = d.r_h1[r], h2 = d.r_h2[r];
            const uint32_t c1 = d.r_c1[r], c2 = d.r_c2[r];
            const bool a2 = h2 > h1;
            const uint64_t ua = cost * (L - (a2 ? h2 : h1)), ub = cost * (L - (a2 ? h1 : h2));
            S.ua[k] = ua;
            S.ub[k] = ub;
            S.thr[k] = (h1 == h2 || ua > slo) ? -1 : (int64_t)(slo - ua);
            S.ab[k] = (a2 ? c2 : c1) | ((a2 ? c1 : c2) << 14) | (uint32_t(a2) << 28) | (uint32_t(h1 != h2) << 29);
            S.nb[k] = d.r_nblk[r];
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
                uint32_t done = __ballot_sync(0xffffffffu, !valid);
                while (done != 0xffffffffu) {
                    const bool ready = !((done >> lane) & 1u) && (conf & ~done) == 0;
                    if (ready) {
                        const uint64_t Wa = W[a], Wb = W[b], Pa = PT[a], Pb = PT[b];
                        const bool pb = Wb < Wa && (int64_t)Wa > thr;
                        const uint32_t ch = pb ? b : a;
                        const uint64_t Pold = pb ? Pb : Pa;
                        W[ch] = pb ? Wb + ub : Wa + ua;
                        PT[ch] = Pold + (uint64_t(S.nb[k]) << 32) + 1;
                        S.Wa[k] = Wa;
                        S.Wb[k] = Wb;
                        S.pt[k] = Pold;
                        S.pickb[k] = pb;
                    }
                    __syncwarp();
                    done |= __ballot_sync(0xffffffffu, ready);
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
            o.chosen[r] = ch;
            o.switched[r] = differ && (int64_t)S.Wa[k] > S.thr[k];
            d.r_final[r] = ch;
            d.r_touchoff[r] = S.pt[k] >> 32;          // offset among this batch's records of ch
            const uint32_t slot = (uint32_t)S.pt[k];
            if (slot - d.q_head[ch] >= d.Q) {
                set_err(d.err, DM_ERR_CAPACITY);
                continue;
            }
            QEntry e;
            e.seq = seq0 + r;
            e.work = e.remaining = pb ? S.ub[k] : S.ua[k];
            e.L = d.r_L[r];
            e.c1 = a_is_c2 ? b : a;
            e.c2 = a_is_c2 ? a : b;
            e.h1 = d.r_h1[r];
            e.h2 = d.r_h2[r];
            e.moved = 0;
            d.q[uint64_t(ch) * d.Q + (slot & (d.Q - 1))] = e;
        }
    }
    __syncthreads();
    for (uint32_t i = threadIdx.x; i < d.M; i += blockDim.x) {
        d.W[i] = W[i];
        d.q_tail[i] = (uint32_t)PT[i];
        d.log_adv[i] = PT[i] >> 32;
    }
    if (threadIdx.x == 0) d.info->final_dirty = 0;
}

cudaError_t launch_choice(const DevState &d, const dm_route_out &o, uint32_t n, uint64_t seq0,
                          cudaStream_t st) {
    if (n == 0) return cudaSuccess;
    const size_t smem = choice_smem(d.M);
    static size_t configured = 0;
    if (smem > configured) {
        cudaError_t e = cudaFuncSetAttribute(k_choice, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             (int)smem);
        if (e != cudaSuccess) return e;
        configured = smem;
    }
    DM_TRY(launch_pdl(k_choice, 1, 1024, smem, st, d, o, n, seq0));
    return cudaGetLastError();
}

}  // namespace dm
