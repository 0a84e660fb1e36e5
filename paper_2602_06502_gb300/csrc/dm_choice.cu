// dm_choice.cu -- queue draining and the SLO-aware choice (Sec. 3.2;
// App. A.1.1: TTFT(r,i) = T_q(r,i) + T_c(r,i)).
//
// Queues: instance i owns a ring buffer of Q entries with monotonically
// increasing head/tail counters; W[i] is the sum of remaining work.
//
// Choice: the decision for a request depends on the loads left by every
// earlier request of the batch, so one CTA walks the batch in arrival order
// with W in shared memory; everything that does not depend on W (uncached
// work, which candidate has more hits) is precomputed in parallel, and the
// queue writes and outputs are emitted in parallel afterwards.
#include "dm_internal.cuh"

namespace dm {

// One warp per instance: run `delta` us of work off the queue head.
__global__ void k_drain(DevState d, uint64_t delta) {
    if (has_err(d.err)) return;
    const int lane = threadIdx.x & 31;
    const uint32_t i = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    if (i >= d.M) return;
    uint32_t head = d.q_head[i];
    const uint32_t tail = d.q_tail[i];
    if (head == tail) return;
    const QEntry *qb = d.q + uint64_t(i) * d.Q;
    uint64_t left = delta, used = 0;
    while (head != tail) {
        const uint32_t cnt = min(32u, tail - head);
        const uint32_t idx = (head + lane) & (d.Q - 1);
        const uint64_t rem = (uint32_t)lane < cnt ? qb[idx].remaining : 0;
        const uint64_t inc = warp_incl_scan(rem, lane);
        const uint32_t done = __ballot_sync(0xffffffffu, (uint32_t)lane < cnt && inc <= left);
        const uint32_t ndone = __popc(done);   // a prefix of the lanes
        if (ndone == cnt) {                    // whole chunk drained
            const uint64_t tot = shfl_u64(inc, 31);
            left -= tot;
            used += tot;
            head += cnt;
            continue;
        }
        const uint64_t before = ndone ? shfl_u64(inc, ndone - 1) : 0;
        if ((uint32_t)lane == ndone) {
            const uint64_t take = left - before;   // < rem of this entry
            d.q[uint64_t(i) * d.Q + idx].remaining = rem - take;
        }
        used += left;
        left = 0;
        head += ndone;
        break;
    }
    if (lane == 0) {
        d.q_head[i] = head;
        d.W[i] -= used;
    }
}

cudaError_t launch_drain(const DevState &d, uint64_t delta, cudaStream_t st) {
    const uint32_t warps = 8;
    k_drain<<<(d.M + warps - 1) / warps, warps * 32, 0, st>>>(d, delta);
    return cudaGetLastError();
}

constexpr uint32_t kChoiceChunk = 512;

// Single CTA (1024 threads).  Dynamic shared memory: W[M] (u64), tail[M] (u32).
__global__ void __launch_bounds__(1024) k_choice(DevState d, dm_route_out o, uint32_t n, uint64_t seq0) {
    extern __shared__ __align__(16) unsigned char smem[];
    __shared__ uint32_t s_c1[kChoiceChunk], s_c2[kChoiceChunk];
    __shared__ uint64_t s_u1[kChoiceChunk], s_u2[kChoiceChunk];
    __shared__ uint8_t s_cls[kChoiceChunk];      // 0: equal hits, 1: c1 has more, 2: c2 has more
    __shared__ uint32_t s_ch[kChoiceChunk], s_slot[kChoiceChunk];
    __shared__ uint64_t s_t1[kChoiceChunk], s_t2[kChoiceChunk];
    __shared__ uint8_t s_sw[kChoiceChunk];
    if (has_err(d.err)) return;
    uint64_t *W = reinterpret_cast<uint64_t *>(smem);
    uint32_t *tail = reinterpret_cast<uint32_t *>(W + d.M);
    for (uint32_t i = threadIdx.x; i < d.M; i += blockDim.x) {
        W[i] = d.W[i];
        tail[i] = d.q_tail[i];
    }
    const uint64_t cost = d.cost, slo = d.slo;
    for (uint32_t base = 0; base < n; base += kChoiceChunk) {
        const uint32_t m = min(kChoiceChunk, n - base);
        __syncthreads();
        for (uint32_t k = threadIdx.x; k < m; k += blockDim.x) {
            const uint32_t r = base + k;
            const uint32_t L = d.r_L[r], h1 = d.r_h1[r], h2 = d.r_h2[r];
            s_c1[k] = d.r_c1[r];
            s_c2[k] = d.r_c2[r];
            s_u1[k] = cost * (L - h1);
            s_u2[k] = cost * (L - h2);
            s_cls[k] = h1 == h2 ? 0 : (h1 > h2 ? 1 : 2);
        }
        __syncthreads();
        if (threadIdx.x == 0) {
            for (uint32_t k = 0; k < m; ++k) {
                const uint32_t c1 = s_c1[k], c2 = s_c2[k];
                const uint64_t W1 = W[c1], W2 = W[c2];
                const uint64_t u1 = s_u1[k], u2 = s_u2[k];
                const uint32_t cls = s_cls[k];
                const uint64_t t1 = W1 + u1, t2 = W2 + u2;
                bool pick2;
                uint8_t sw = 0;
                if (cls == 0) {
                    pick2 = W2 < W1;
                } else {
                    const bool a2 = cls == 2;          // a = higher-hit candidate
                    const uint64_t ta = a2 ? t2 : t1;
                    const uint64_t Wa = a2 ? W2 : W1, Wb = a2 ? W1 : W2;
                    if (ta <= slo) {
                        pick2 = a2;
                    } else {
                        sw = 1;
                        pick2 = (Wb < Wa) ? !a2 : a2;
                    }
                }
                const uint32_t ch = pick2 ? c2 : c1;
                W[ch] = (pick2 ? W2 : W1) + (pick2 ? u2 : u1);
                s_ch[k] = ch;
                s_slot[k] = tail[ch]++;
                s_t1[k] = t1;
                s_t2[k] = t2;
                s_sw[k] = sw;
            }
        }
        __syncthreads();
        for (uint32_t k = threadIdx.x; k < m; k += blockDim.x) {
            const uint32_t r = base + k;
            const uint32_t ch = s_ch[k];
            const bool pick2 = ch == s_c2[k];
            o.ttft1[r] = s_t1[k];
            o.ttft2[r] = s_t2[k];
            o.chosen[r] = ch;
            o.switched[r] = s_sw[k];
            d.r_final[r] = ch;
            const uint32_t slot = s_slot[k];
            if (slot - d.q_head[ch] >= d.Q) {
                set_err(d.err, DM_ERR_CAPACITY);
                continue;
            }
            QEntry e;
            e.seq = seq0 + r;
            e.work = e.remaining = pick2 ? s_u2[k] : s_u1[k];
            e.L = d.r_L[r];
            e.c1 = s_c1[k];
            e.c2 = s_c2[k];
            e.h1 = d.r_h1[r];
            e.h2 = d.r_h2[r];
            e.moved = 0;
            d.q[uint64_t(ch) * d.Q + (slot & (d.Q - 1))] = e;
        }
    }
    __syncthreads();
    for (uint32_t i = threadIdx.x; i < d.M; i += blockDim.x) {
        d.W[i] = W[i];
        d.q_tail[i] = tail[i];
    }
}

cudaError_t launch_choice(const DevState &d, const dm_route_out &o, uint32_t n, uint64_t seq0,
                          cudaStream_t st) {
    if (n == 0) return cudaSuccess;
    const size_t smem = size_t(d.M) * (sizeof(uint64_t) + sizeof(uint32_t));
    static size_t configured = 0;
    if (smem > configured) {
        cudaError_t e = cudaFuncSetAttribute(k_choice, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             (int)smem);
        if (e != cudaSuccess) return e;
        configured = smem;
    }
    k_choice<<<1, 1024, smem, st>>>(d, o, n, seq0);
    return cudaGetLastError();
}

}  // namespace dm
