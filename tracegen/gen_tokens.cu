// gen_tokens.cu -- device twin of tracegen.trace.piece_tokens: fills a token
// buffer from piece descriptors with the counter-based generator
//   token(stream, pos) = mix64(token_seed ^ stream * PHI ^ pos) mod vocab,
// mix64 being one SplitMix64 output step.  Input generation only.
#include <cstdint>
#include <cuda_runtime.h>

namespace {

__device__ __forceinline__ uint64_t mix64(uint64_t x) {
    uint64_t z = x + 0x9E3779B97F4A7C15ULL;
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
    return z ^ (z >> 31);
}

// One CTA per piece (grid-stride over pieces), threads over its positions.
__global__ void k_fill(uint32_t *dst, const uint64_t *p_dst, const uint64_t *p_stream, const uint64_t *p_start,
                       const uint32_t *p_len, uint64_t n_pieces, uint64_t seed, uint64_t vocab) {
    for (uint64_t p = blockIdx.x; p < n_pieces; p += gridDim.x) {
        const uint64_t base = seed ^ (p_stream[p] * 0x9E3779B97F4A7C15ULL);
        uint32_t *out = dst + p_dst[p];
        const uint64_t s0 = p_start[p];
        const uint32_t len = p_len[p];
        for (uint32_t k = threadIdx.x; k < len; k += blockDim.x)
            out[k] = (uint32_t)(mix64(base ^ (s0 + k)) % vocab);
    }
}

}  // namespace

extern "C" int tg_fill_tokens(uint32_t *dst, const uint64_t *p_dst, const uint64_t *p_stream,
                              const uint64_t *p_start, const uint32_t *p_len, uint64_t n_pieces, uint64_t seed,
                              uint64_t vocab, void *stream) {
    if (n_pieces == 0) return 0;
    const uint64_t grid = n_pieces < 65535 * 4 ? n_pieces : 65535 * 4;
    k_fill<<<(unsigned)grid, 256, 0, (cudaStream_t)stream>>>(dst, p_dst, p_stream, p_start, p_len, n_pieces, seed,
                                                              vocab);
    return (int)cudaGetLastError();
}
