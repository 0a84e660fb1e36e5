// dm_potc.cu -- the power-of-d-choices experiment behind DualMap's choice of
// two candidates (App. A.8, "Optimal Candidate Set Size"): m balls into n
// bins, each ball to the least loaded of d uniformly random bins (ties to
// the earlier choice), the maximum bin load of each trial.
//
// Ball t's choice k in trial s uses counter c = (s * m + t) * d + k: the
// (c+1)-th output of SplitMix64 (Steele, Lea & Flood 2014) seeded with
// `seed`, scaled to a bin as floor(x * n / 2^64).
//
// One thread per trial; its n bin loads live in a shared-memory column
// (bin b of thread j at [b * blockDim + j], so a warp's accesses to any
// bins fall in distinct banks).
#include "dm_internal.cuh"

namespace dm {

__device__ __forceinline__ uint32_t potc_choice(uint64_t seed, uint64_t c, uint32_t n) {
    const uint64_t x = splitmix_step(seed + c * 0x9E3779B97F4A7C15ull);   // state after c increments
    return (uint32_t)__umul64hi(x, n);
}

__global__ void k_potc(uint32_t n, uint64_t m, uint32_t d, uint32_t trials, uint64_t seed, uint32_t *max_load) {
    extern __shared__ uint32_t s_load[];
    const uint32_t T = blockDim.x;
    uint32_t *L = s_load + threadIdx.x;
    const uint32_t s = blockIdx.x * T + threadIdx.x;
    if (s >= trials) return;
    for (uint32_t b = 0; b < n; ++b) L[b * T] = 0;
    for (uint64_t t = 0; t < m; ++t) {
        const uint64_t c0 = (uint64_t(s) * m + t) * d;
        uint32_t best = potc_choice(seed, c0, n), bl = L[best * T];
        for (uint32_t k = 1; k < d; ++k) {
            const uint32_t b = potc_choice(seed, c0 + k, n), l = L[b * T];
            if (l < bl) { best = b; bl = l; }
        }
        L[best * T] = bl + 1;
    }
    uint32_t mx = 0;
    for (uint32_t b = 0; b < n; ++b) mx = max(mx, L[b * T]);
    max_load[s] = mx;
}

}  // namespace dm

extern "C" dm_status dm_potc_max_loads(uint32_t n_bins, uint64_t m_balls, uint32_t d, uint32_t trials,
                                       uint64_t seed, uint32_t *max_load_dev, void *stream) {
    if (n_bins < 1 || n_bins > 256 || d < 1 || d > 64 || m_balls > 0xFFFFFFFFull || !max_load_dev)
        return DM_ERR_INVALID_ARG;
    if (trials == 0) return DM_OK;
    // 64 trials per block (32 when 48 KB of loads allow no more): each
    // trial is one long dependent chain, so spreading the trials over the
    // SMs matters more than filling any one of them
    uint32_t T = (48u * 1024u) / (4u * n_bins);
    T = T > 64 ? 64 : T;
    T = T / 32 * 32;
    const unsigned grid = (trials + T - 1) / T;
    dm::k_potc<<<grid, T, size_t(T) * n_bins * 4, static_cast<cudaStream_t>(stream)>>>(n_bins, m_balls, d, trials,
                                                                                        seed, max_load_dev);
    return cudaGetLastError() == cudaSuccess ? DM_OK : DM_ERR_CUDA;
}
