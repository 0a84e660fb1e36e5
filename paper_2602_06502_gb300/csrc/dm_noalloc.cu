// dm_noalloc.cu -- dm_hash_prompts_noalloc: prompt hashing (block keys and
// ring positions, the same values as dm_hash_prompts) for callers that must
// not allocate device memory.  Its scratch is a fixed array in this file;
// the caller's key buffer holds the per-block prefix values until they are
// turned into keys in place.
#include <mutex>

#include "dm_internal.cuh"

namespace dm {
namespace {

constexpr uint32_t kNaReq = DM_NOALLOC_MAX_REQUESTS;
constexpr uint64_t kNaBlocks = DM_NOALLOC_MAX_BLOCKS;
constexpr uint64_t kNaSegs = kNaBlocks / kSegBlocks + kNaReq;

constexpr size_t align256(size_t x) { return (x + 255) / 256 * 256; }

// Byte offsets of the scratch arrays.
constexpr size_t kOffL = 0;
constexpr size_t kOffNblk = kOffL + align256(4 * kNaReq);
constexpr size_t kOffSegoff = kOffNblk + align256(4 * kNaReq);
constexpr size_t kOffTokoff = kOffSegoff + align256(4 * kNaReq);
constexpr size_t kOffBlkoff = kOffTokoff + align256(8 * kNaReq);
constexpr size_t kOffSegReq = kOffBlkoff + align256(8 * kNaReq);
constexpr size_t kOffSegTot = kOffSegReq + align256(4 * kNaSegs);
constexpr size_t kOffSegTot2 = kOffSegTot + align256(8 * kNaSegs);
constexpr size_t kOffSegCarry = kOffSegTot2 + align256(8 * kNaSegs);
constexpr size_t kOffInfo = kOffSegCarry + align256(8 * kNaSegs);
constexpr size_t kOffErr = kOffInfo + align256(sizeof(BatchInfo));
constexpr size_t kScratchBytes = kOffErr + 256;

// Shared by every call on a device; holds the last call's contents.
static __device__ __align__(256) unsigned char g_na_scratch[kScratchBytes];

constexpr int kMaxDevices = 64;
std::mutex g_na_mutex;
unsigned char *g_na_addr[kMaxDevices] = {};

// Device address of the scratch array for the current device (looked up once
// per device, with that device current).
cudaError_t scratch_address(unsigned char **out) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lock(g_na_mutex);
    if (!g_na_addr[dev]) {
        void *p = nullptr;
        e = cudaGetSymbolAddress(&p, g_na_scratch);
        if (e != cudaSuccess) return e;
        g_na_addr[dev] = static_cast<unsigned char *>(p);
    }
    *out = g_na_addr[dev];
    return cudaSuccess;
}

uint64_t na_splitmix_next(uint64_t &s) {
    uint64_t z = (s += 0x9E3779B97F4A7C15ULL);
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
    return z ^ (z >> 31);
}

// Warp per request: ring positions from the prefix values, then the prefix
// values in the caller's buffer become cache keys in place.
__global__ void k_na_finish(DevState d, uint32_t n, uint64_t *keys, uint64_t *key_off, uint64_t *pos) {
    if (has_err(d.err)) return;
    const int lane = threadIdx.x & 31;
    const uint32_t r = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    if (r >= n) return;
    request_carries(d, r, lane);
    __syncwarp();
    uint64_t p1, p2;
    route_positions(d, r, lane, p1, p2);   // reads the prefix value of block K-1
    __syncwarp();
    const uint32_t nblk = d.r_nblk[r], s0 = d.r_segoff[r];
    const uint64_t bo = d.r_blkoff[r];
    for (uint32_t b = lane; b < nblk; b += 32)
        keys[bo + b] = cache_key(keys[bo + b] + d.seg_carry[s0 + b / kSegBlocks], d.Sc);
    if (lane == 0) {
        key_off[r] = bo;
        pos[2 * r] = p1;
        pos[2 * r + 1] = p2;
        if (r == n - 1) key_off[n] = bo + nblk;
    }
}

}  // namespace
}  // namespace dm

extern "C" DM_API dm_status dm_hash_prompts_noalloc(uint32_t block_tokens, uint32_t route_prefix_blocks,
                                                    uint64_t seed, const dm_batch *b, uint64_t *keys_dev,
                                                    uint64_t *key_off_dev, uint64_t *pos_dev, void *stream) {
    using namespace dm;
    const uint32_t B = block_tokens;
    if (!(B == 4 || B == 8 || B == 16 || B == 32 || B == 64)) return DM_ERR_INVALID_ARG;
    if (route_prefix_blocks < 1 || route_prefix_blocks > kMaxRouteBlocks) return DM_ERR_INVALID_ARG;
    if (!b || b->reserved0) return DM_ERR_INVALID_ARG;
    if (b->n == 0) return DM_OK;
    if (!b->tokens || !b->offsets || !b->lengths || !keys_dev || !key_off_dev || !pos_dev)
        return DM_ERR_INVALID_ARG;
    if (reinterpret_cast<uintptr_t>(b->tokens) & 15) return DM_ERR_INVALID_ARG;
    if (b->n > kNaReq || b->total_tokens / B > kNaBlocks) return DM_ERR_CAPACITY;

    unsigned char *base = nullptr;
    cudaError_t e = scratch_address(&base);
    if (e != cudaSuccess) return DM_ERR_CUDA;
    cudaStream_t st = static_cast<cudaStream_t>(stream);

    DevState d{};
    d.B = B;
    d.Kroute = route_prefix_blocks;
    d.Kf2 = route_prefix_blocks;   // fixed hash length: f2 over the first K_route blocks
    d.ad_step = 0;
    d.max_batch = kNaReq;
    d.max_blocks = kNaBlocks;
    d.max_segs = kNaSegs;
    uint64_t s = seed;   // same key material as dm_create with this seed
    for (uint32_t j = 0; j < B; ++j) d.K1[j] = (uint32_t)na_splitmix_next(s);
    for (uint32_t j = 0; j < B; ++j) d.K2[j] = (uint32_t)na_splitmix_next(s);
    d.G1 = na_splitmix_next(s) | 1ull;
    d.G2 = na_splitmix_next(s) | 1ull;
    d.Sc = na_splitmix_next(s);
    d.Sr1 = na_splitmix_next(s);
    d.Sr2 = na_splitmix_next(s);
    d.Sv1 = na_splitmix_next(s);
    d.Sv2 = na_splitmix_next(s);
    d.r_L = reinterpret_cast<uint32_t *>(base + kOffL);
    d.r_nblk = reinterpret_cast<uint32_t *>(base + kOffNblk);
    d.r_segoff = reinterpret_cast<uint32_t *>(base + kOffSegoff);
    d.r_tokoff = reinterpret_cast<uint64_t *>(base + kOffTokoff);
    d.r_blkoff = reinterpret_cast<uint64_t *>(base + kOffBlkoff);
    d.seg_req = reinterpret_cast<uint32_t *>(base + kOffSegReq);
    d.seg_total = reinterpret_cast<uint64_t *>(base + kOffSegTot);
    d.seg_total2 = reinterpret_cast<uint64_t *>(base + kOffSegTot2);
    d.seg_carry = reinterpret_cast<uint64_t *>(base + kOffSegCarry);
    d.info = reinterpret_cast<BatchInfo *>(base + kOffInfo);
    d.err = reinterpret_cast<uint32_t *>(base + kOffErr);
    d.plocal = keys_dev;   // prefix values live in the output until converted

    // Only the error word must start at zero: every other scratch entry a
    // kernel reads is written earlier in the same call.
    e = cudaMemsetAsync(d.err, 0, sizeof(uint32_t), st);
    if (e == cudaSuccess) e = launch_setup(d, *b, st);
    if (e == cudaSuccess) e = launch_hash(d, *b, hash_grid_size(), st);
    if (e == cudaSuccess) {
        k_na_finish<<<(b->n + 7) / 8, 256, 0, st>>>(d, b->n, keys_dev, key_off_dev, pos_dev);
        e = cudaGetLastError();
    }
    uint32_t err = 0;
    if (e == cudaSuccess) e = cudaMemcpyAsync(&err, d.err, sizeof(uint32_t), cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
    if (e != cudaSuccess) return DM_ERR_CUDA;
    return static_cast<dm_status>(err);
}
