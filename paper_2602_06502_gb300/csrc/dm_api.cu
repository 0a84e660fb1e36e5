// dm_api.cu -- host side of the C ABI declared in include/dualmap.h:
// argument checks, device memory ownership, stream ordering, error mapping.
// Every computation of the routing path runs in the kernels of the other
// translation units; this file only validates, allocates and enqueues.
#include <cstdio>
#include <algorithm>
#include <atomic>
#include <cstring>
#include <utility>
#include <vector>

#include "dm_internal.cuh"

using dm::DevState;
using dm::QEntry;
using dm::Rec;
using dm::Slot;

struct StageEvent {
    int stage;
    cudaEvent_t a, b;
};

struct dm_handle {
    dm_config cfg{};
    DevState d{};            // main scheduler state (kernel parameter)
    DevState dh{};           // same, with the scratch of dm_hash_prompts
    cudaStream_t st = nullptr;
    std::vector<uint8_t> state;   // host mirror: 0 absent, 1 live, 2 draining
    uint32_t n_live = 0;
    uint64_t seq_next = 0, t_prev = 0;
    bool have_time = false;
    bool pending = false;
    uint32_t pending_n = 0;
    bool shard_open = false;   // between dm_route_shard_begin and dm_route_shard_finish
    uint32_t shard_n = 0;
    uint64_t pending_seq0 = 0;
    uint32_t rebalance_calls = 0;
    int hash_grid = 0;
    uint64_t epoch = 0;   // routing calls so far (the routing kernel's record checks)
    // adaptive prefix length: the second expanded-node table (the next
    // window's target), requests and non-empty batches in the current window
    uint64_t *ad_alt = nullptr;
    uint64_t ad_T = 0;
    uint32_t ad_batches = 0;
    uint64_t *vpos_buf[dm::kMaxD][2] = {};
    uint32_t *owner_buf[dm::kMaxD][2] = {}, *vidx_buf[dm::kMaxD][2] = {};
    int cur[dm::kMaxD] = {};
    uint64_t *ring_spos = nullptr;
    uint32_t *ring_svidx = nullptr;
    std::vector<Slot *> tables;   // the index buffer first allocated for each id (null: never added)
    uint32_t pool_target = 0;     // spare index buffers wanted (one per allocated id, up to rebuild_pool)
    std::vector<Rec *> logs, logs2;        // both log buffers
    std::vector<uint8_t *> stales, stales2;
    std::vector<uint32_t *> homes, homes2;  // both index-home logs
    std::vector<void *> allocs;    // every cudaMalloc of the handle
    // staging of the host-buffer entry points: two buffers, so the upload of
    // one batch (on copy_st) overlaps the routing of the previous one
    struct HostStage {
        uint32_t *tokens = nullptr, *lengths = nullptr;
        uint64_t *offsets = nullptr;
        dm_route_out out{};
        cudaEvent_t copied = nullptr, consumed = nullptr;
        bool used = false;
    } hs[2];
    int hs_next = 0;
    cudaStream_t copy_st = nullptr;
    uint32_t profiling = 0;   // bit s: time stage s
    std::vector<StageEvent> events;
    std::vector<cudaEvent_t> ev_pool;
    double stage_ms[DM_STAGE_COUNT] = {};
    uint64_t stage_calls[DM_STAGE_COUNT] = {};
    dm_status sticky = DM_OK;
    // device staging of dm_rebalance's host results
    dm_migration *rb_out_dev = nullptr;
    uint32_t rb_out_cap = 0;
    uint32_t *rb_n_dev = nullptr;
};

namespace {

// Test hook (dm_test_fail_alloc): the allocation with this ordinal fails.
std::atomic<int64_t> g_fail_at{-1};
std::atomic<int64_t> g_alloc_seq{0};

template <typename T>
cudaError_t dalloc(dm_handle *h, T **p, size_t count) {
    const int64_t fail_at = g_fail_at.load(std::memory_order_relaxed);
    if (fail_at >= 0 && g_alloc_seq.fetch_add(1, std::memory_order_relaxed) == fail_at) {
        *p = nullptr;
        return cudaErrorMemoryAllocation;
    }
    void *q = nullptr;
    cudaError_t e = cudaMalloc(&q, count ? count * sizeof(T) : 16);
    if (e != cudaSuccess) { *p = nullptr; return e; }
    h->allocs.push_back(q);
    *p = static_cast<T *>(q);
    return cudaSuccess;
}

uint64_t pow2_at_least(uint64_t x) {
    uint64_t p = 1;
    while (p < x) p <<= 1;
    return p;
}

dm_status map_cuda(dm_handle *h, cudaError_t e) {
    if (e == cudaSuccess) return DM_OK;
    if (h->sticky == DM_OK) h->sticky = (e == cudaErrorMemoryAllocation) ? DM_ERR_OOM : DM_ERR_CUDA;
    return h->sticky;
}

// Split R into the levels of the 32-ary search tree.
void set_levels(DevState &d, uint32_t R) {
    d.R = R;
    d.lev_n[0] = R;
    uint32_t k = 0;
    while (d.lev_n[k] > 32 && k + 1 < (uint32_t)dm::kMaxLevels) {
        d.lev_n[k + 1] = (d.lev_n[k] + 31) / 32;
        ++k;
    }
    d.nlev = k + 1;
    d.lev_off[1] = 0;
    for (uint32_t j = 1; j + 1 < d.nlev; ++j) d.lev_off[j + 1] = d.lev_off[j] + d.lev_n[j];
}

// Events come from a pool that dm_get_stage_times refills, so timing a
// stage costs two cudaEventRecord calls.
cudaEvent_t pool_event(dm_handle *h) {
    if (h->ev_pool.empty()) {
        cudaEvent_t e = nullptr;
        if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
        return e;
    }
    cudaEvent_t e = h->ev_pool.back();
    h->ev_pool.pop_back();
    return e;
}

struct Stage {
    dm_handle *h;
    int s;
    cudaEvent_t a = nullptr, b = nullptr;
    Stage(dm_handle *h_, int s_) : h(h_), s(s_) {
        if (!(h->profiling >> s & 1u)) return;
        a = pool_event(h);
        b = pool_event(h);
        if (a && b) cudaEventRecord(a, h->st);
    }
    ~Stage() {
        if (a && b) {
            cudaEventRecord(b, h->st);
            h->events.push_back(StageEvent{s, a, b});
        } else {
            if (a) h->ev_pool.push_back(a);
            if (b) h->ev_pool.push_back(b);
        }
    }
};

uint64_t splitmix_next(uint64_t &s) {
    uint64_t z = (s += 0x9E3779B97F4A7C15ULL);
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
    return z ^ (z >> 31);
}

dm_status check_live(dm_handle *h) {
    if (!h) return DM_ERR_INVALID_ARG;
    return h->sticky;
}

// Read-only introspection keeps working after a sticky error.
dm_status check_handle(dm_handle *h) {
    return h ? DM_OK : DM_ERR_INVALID_ARG;
}

}  // namespace

extern "C" {

const char *dm_status_string(dm_status s) {
    switch (s) {
        case DM_OK: return "ok";
        case DM_ERR_INVALID_ARG: return "invalid argument";
        case DM_ERR_CAPACITY: return "capacity exceeded";
        case DM_ERR_NO_INSTANCES: return "fewer than two live instances";
        case DM_ERR_DUPLICATE_ID: return "instance id already live or still draining";
        case DM_ERR_UNKNOWN_ID: return "instance id not live";
        case DM_ERR_ORDER: return "batch time earlier than the previous batch";
        case DM_ERR_CUDA: return "CUDA runtime error";
        case DM_ERR_TIMEOUT: return "bounded device loop gave up";
        case DM_ERR_OOM: return "out of memory";
        case DM_ERR_BOUNDS: return "a device index check failed (debug build)";
    }
    return "unknown status";
}

void dm_destroy(dm_handle *h) {
    if (!h) return;
    cudaStreamSynchronize(h->st);
    if (h->copy_st) {
        cudaStreamSynchronize(h->copy_st);
        cudaStreamDestroy(h->copy_st);
    }
    for (auto &x : h->hs) {
        if (x.copied) cudaEventDestroy(x.copied);
        if (x.consumed) cudaEventDestroy(x.consumed);
    }
    for (auto &ev : h->events) { cudaEventDestroy(ev.a); cudaEventDestroy(ev.b); }
    for (auto e : h->ev_pool) cudaEventDestroy(e);
    for (void *p : h->allocs) cudaFree(p);
    delete h;
}

dm_status dm_create(const dm_config *cfg, dm_handle **out) {
    if (!cfg || !out) return DM_ERR_INVALID_ARG;
    *out = nullptr;
    const dm_config &c = *cfg;
    const uint32_t B = c.block_tokens;
    if (!(B == 4 || B == 8 || B == 16 || B == 32 || B == 64)) return DM_ERR_INVALID_ARG;
    if (c.route_prefix_blocks < 1 || c.route_prefix_blocks > dm::kMaxRouteBlocks) return DM_ERR_INVALID_ARG;
    if (c.vnodes_per_instance < 1 || c.vnodes_per_instance > 65536) return DM_ERR_INVALID_ARG;
    if (c.max_instances < 2 || c.max_instances > dm::kMaxInstances) return DM_ERR_INVALID_ARG;
    if (uint64_t(c.max_instances) * c.vnodes_per_instance > (1ull << 31)) return DM_ERR_INVALID_ARG;
    if (c.cache_capacity_blocks < 1 || c.cost_us_per_token < 1 || c.hot_den < 1) return DM_ERR_INVALID_ARG;
    if (c.max_batch < 1 || c.max_batch > (1u << 24) || c.max_batch_tokens < B) return DM_ERR_INVALID_ARG;
    if (c.max_queue && (c.max_queue & (c.max_queue - 1))) return DM_ERR_INVALID_ARG;
    if (c.index_slots_log2 > 32) return DM_ERR_INVALID_ARG;   // index homes are logged as u32
    if (c.choice_rule > DM_RULE_PREBLE) return DM_ERR_INVALID_ARG;
    if (c.rebalance_flags > (DM_REBALANCE_SLO_TARGET | DM_REBALANCE_DOUBLE_OVERLOAD | DM_REBALANCE_FRESH_HITS))
        return DM_ERR_INVALID_ARG;
    if ((c.rebalance_flags & DM_REBALANCE_FRESH_HITS) &&   // keys are queued by the pair-rule choice kernel
        (!c.rebalance_key_blocks || c.rebalance_key_blocks > (1ull << 40) || c.choice_rule >= DM_RULE_LEAST_LOADED ||
         (c.candidates && c.candidates != 2)))
        return DM_ERR_INVALID_ARG;
    if (c.candidates > dm::kMaxD) return DM_ERR_INVALID_ARG;
    if (c.candidates && c.candidates != 2 && (c.choice_rule != DM_RULE_DUALMAP || c.adapt_step_blocks))
        return DM_ERR_INVALID_ARG;
    if (c.adapt_step_blocks &&
        (c.adapt_max_blocks <= c.route_prefix_blocks || c.adapt_max_blocks > 2048 || c.adapt_window < 1))
        return DM_ERR_INVALID_ARG;

    dm_handle *h = new dm_handle();
    h->cfg = c;
    h->st = static_cast<cudaStream_t>(c.stream);
    DevState &d = h->d;
    d.B = B;
    d.Kroute = c.route_prefix_blocks;
    d.V = c.vnodes_per_instance;
    d.M = c.max_instances;
    d.C = c.cache_capacity_blocks;
    d.slo = c.slo_us;
    d.cost = c.cost_us_per_token;
    d.hot_num = c.hot_num;
    d.hot_den = c.hot_den;
    d.max_batch = c.max_batch;
    d.rule = c.choice_rule;
    d.rb_flags = c.rebalance_flags;
    d.ad_step = c.adapt_step_blocks;
    d.ad_max = c.adapt_step_blocks ? c.adapt_max_blocks : c.route_prefix_blocks;
    d.Kf2 = d.ad_max;
    d.loop_limit = c.test_loop_limit;
    d.max_blocks = c.max_batch_tokens / B;
    d.max_segs = d.max_blocks / dm::kSegBlocks + c.max_batch;
    if (d.max_segs >= (1ull << 31)) {   // segment counts and offsets are 32-bit
        delete h;
        return DM_ERR_INVALID_ARG;
    }
    // routing order: a head long enough for the longest routing prefix
    d.Ccols = (d.Kf2 + dm::kSegBlocks - 1) / dm::kSegBlocks;
    d.H = std::max<uint32_t>(dm::kHeadSegs, d.Ccols);
    d.T = c.max_touch_per_instance ? c.max_touch_per_instance : d.max_blocks;
    d.S = pow2_at_least(2 * (d.C + d.T));
    if (c.index_slots_log2 && (1ull << c.index_slots_log2) > d.S) d.S = 1ull << c.index_slots_log2;
    if (d.S < 64) d.S = 64;   // at least a few whole groups
    if (d.S > (1ull << 32)) {
        delete h;
        return DM_ERR_INVALID_ARG;
    }
    // Rebuild threshold: a quarter of the slots when that still holds C + T
    // keys (evicted keys keep their slots, and fuller buckets lengthen probes
    // and touches: measured 5.6 % faster than half on the long-context
    // bench), else half.
    d.rb_thr = d.S / 4 >= d.C + d.T ? d.S / 4 : d.S / 2;
    // a pool smaller than the instance count makes rebuilds wait up to
    // ceil(M / pool) commits: the index must hold that many commits' touches
    // above half full
    h->pool_target = c.rebuild_pool && c.rebuild_pool < c.max_instances ? c.rebuild_pool : c.max_instances;
    if (h->pool_target < c.max_instances &&
        d.S / 2 < uint64_t((c.max_instances + h->pool_target - 1) / h->pool_target) * d.T) {
        delete h;
        return DM_ERR_INVALID_ARG;
    }
    d.logcap = pow2_at_least(2 * (d.C + d.T));
    if (d.logcap < 1024) d.logcap = 1024;   // whole 16-byte flag groups (eviction reads flags 16 at a time)
    d.Q = c.max_queue ? c.max_queue : 65536;
    d.rb_cap = (uint32_t)pow2_at_least(d.Q > d.M ? d.Q : d.M);
    // key material: SplitMix64(seed) -> K1[0..B), K2[0..B), G1|1, G2|1, Sc, Sr1, Sr2, Sv1, Sv2
    uint64_t s = c.seed;
    for (uint32_t j = 0; j < B; ++j) d.K1[j] = (uint32_t)splitmix_next(s);
    for (uint32_t j = 0; j < B; ++j) d.K2[j] = (uint32_t)splitmix_next(s);
    d.G1 = splitmix_next(s) | 1ull;
    d.G2 = splitmix_next(s) | 1ull;
    d.Sc = splitmix_next(s);
    d.Sr1 = splitmix_next(s);
    d.Sr2 = splitmix_next(s);
    d.Sv1 = splitmix_next(s);
    d.Sv2 = splitmix_next(s);
    // functions 3..kMaxD of the d-candidate path, drawn after DualMap's
    uint32_t kx[dm::kMaxD - 2][64] = {};
    for (uint32_t f = 0; f + 2 < dm::kMaxD; ++f) {
        for (uint32_t j = 0; j < B; ++j) kx[f][j] = (uint32_t)splitmix_next(s);
        d.Gx[f] = splitmix_next(s) | 1ull;
        d.Srx[f] = splitmix_next(s);
        d.Svx[f] = splitmix_next(s);
    }
    d.nrings = c.candidates > 2 ? c.candidates : 2;
    d.nd = c.candidates ? c.candidates : 2;

    const uint64_t M = d.M, Rmax = M * d.V;
    cudaError_t e = cudaSuccess;
    auto A = [&](cudaError_t x) { if (e == cudaSuccess) e = x; };
    for (uint32_t f = 0; f < d.nrings; ++f)
        for (int b = 0; b < 2; ++b) {
            A(dalloc(h, &h->vpos_buf[f][b], Rmax));
            A(dalloc(h, &h->owner_buf[f][b], Rmax));
            A(dalloc(h, &h->vidx_buf[f][b], Rmax));
        }
    uint64_t tree_n = 0;
    for (uint64_t n = Rmax; n > 32;) { n = (n + 31) / 32; tree_n += n; }
    for (uint32_t f = 0; f < d.nrings; ++f) A(dalloc(h, &d.ring[f].tree, tree_n + 32));
    uint32_t P = 1;
    while (P < d.V) P <<= 1;
    A(dalloc(h, &h->ring_spos, uint64_t(d.nrings) * P));
    A(dalloc(h, &h->ring_svidx, uint64_t(d.nrings) * P));
    uint32_t *kx_dev = nullptr;
    A(dalloc(h, &kx_dev, (dm::kMaxD - 2) * 64));
    d.Kx = kx_dev;
    A(dalloc(h, &d.rd_cand, uint64_t(c.max_batch) * d.nd));
    A(dalloc(h, &d.rd_hit, uint64_t(c.max_batch) * d.nd));
    A(dalloc(h, &d.inst_state, M));
    A(dalloc(h, &d.next_live, M));
    A(dalloc(h, &d.W, M));
    A(dalloc(h, &d.q_head, M));
    A(dalloc(h, &d.q_tail, M));
    A(dalloc(h, &d.q, M * d.Q));
    A(dalloc(h, &d.table, M));
    A(dalloc(h, &d.logbuf, M));
    A(dalloc(h, &d.table_alt, M));
    A(dalloc(h, &d.pool, h->pool_target));
    A(dalloc(h, &d.rb_slot, M));
    A(dalloc(h, &d.rb_rr, 1));
    A(dalloc(h, &d.logbuf_alt, M));
    A(dalloc(h, &d.stale, M));
    A(dalloc(h, &d.stale_alt, M));
    A(dalloc(h, &d.loghome, M));
    A(dalloc(h, &d.loghome_alt, M));
    A(dalloc(h, &d.mt_flags, M));
    A(dalloc(h, &d.mt_newtail, M));
    A(dalloc(h, &d.mc_chunk_off, M + 1));
    A(dalloc(h, &d.mr_chunk_off, M + 1));
    d.mc_cap = M * (d.logcap / dm::kEvChunk + 1);
    A(dalloc(h, &d.mc_chunk_live, d.mc_cap));
    A(dalloc(h, &d.log_front, M));
    A(dalloc(h, &d.log_tail, M));
    A(dalloc(h, &d.live, M));
    A(dalloc(h, &d.used, M));
    A(dalloc(h, &d.log_adv, M));
    A(dalloc(h, &d.log_base, M));
    A(dalloc(h, &d.clock, 1));
    A(dalloc(h, &d.maint_count, 2));
    A(dalloc(h, &d.err, 1));
    A(dalloc(h, &d.seq_next, 1));
    A(dalloc(h, &d.metrics, 1));
    uint64_t ad_levels = 0;
    if (c.adapt_step_blocks) {
        // at most n expanded nodes per level (each holds >= 1/n of a window's requests)
        ad_levels = (d.ad_max - c.route_prefix_blocks + d.ad_step - 1) / d.ad_step + 1;
        d.ad_set_mask = pow2_at_least(std::max<uint64_t>(1024, 4 * M * ad_levels)) - 1;
        d.ad_cnt_mask = pow2_at_least(std::max<uint64_t>(1024, 2ull * c.max_batch * c.adapt_window * ad_levels)) - 1;
        if (d.ad_cnt_mask >= (1ull << 26)) {
            dm_destroy(h);
            return DM_ERR_INVALID_ARG;
        }
        A(dalloc(h, &d.ad_set, d.ad_set_mask + 1));
        A(dalloc(h, &h->ad_alt, d.ad_set_mask + 1));
        A(dalloc(h, &d.ad_cnt, d.ad_cnt_mask + 1));
    }
    if (c.choice_rule >= DM_RULE_LEAST_LOADED) A(dalloc(h, &d.h_all, uint64_t(c.max_batch) * M));
    A(dalloc(h, &d.rb_key, d.rb_cap));
    A(dalloc(h, &d.rb_seq, d.rb_cap));
    A(dalloc(h, &d.rb_ttft, d.rb_cap));
    A(dalloc(h, &d.rb_pos, d.rb_cap));
    if (c.rebalance_flags & DM_REBALANCE_FRESH_HITS) {   // queued requests' keys, for fresh rebalancing probes
        d.KQ = pow2_at_least(c.rebalance_key_blocks);
        A(dalloc(h, &d.kring, M * d.KQ));
        A(dalloc(h, &d.kr_head, M));
        A(dalloc(h, &d.kr_tail, M));
        A(dalloc(h, &d.r_koff, c.max_batch));
        A(dalloc(h, &d.rb_hq, d.Q));
    }
    A(dalloc(h, &d.r_hoff, c.max_batch));
    A(dalloc(h, &d.r_toff, c.max_batch));
    A(dalloc(h, &d.seg_pub, d.max_segs));
    A(dalloc(h, &d.r_m1, c.max_batch));
    A(dalloc(h, &d.r_m2, c.max_batch));
    A(dalloc(h, &d.fix_list, c.max_batch));   // every route task at most once
    A(dalloc(h, &d.defer, d.max_segs * dm::kSegBlocks));
    // two sets of batch scratch: routing and dm_hash_prompts
    for (DevState *x : {&h->d, &h->dh}) {
        if (x == &h->dh) {
            const DevState keep = h->d;
            *x = keep;
        }
        A(dalloc(h, &x->r_L, c.max_batch));
        A(dalloc(h, &x->r_nblk, c.max_batch));
        A(dalloc(h, &x->r_segoff, c.max_batch));
        A(dalloc(h, &x->r_tokoff, c.max_batch));
        A(dalloc(h, &x->r_blkoff, c.max_batch));
        A(dalloc(h, &x->seg_req, d.max_segs));
        A(dalloc(h, &x->seg_total, d.max_segs));
        A(dalloc(h, &x->seg_carry, d.max_segs));
        A(dalloc(h, &x->seg_total2, d.max_segs));
        A(dalloc(h, &x->plocal, d.max_blocks));
        if (x == &h->d && c.adapt_step_blocks) A(dalloc(h, &x->p2local, d.max_blocks));
        A(dalloc(h, &x->r_K, c.max_batch));
        A(dalloc(h, &x->r_c1, c.max_batch));
        A(dalloc(h, &x->r_c2, c.max_batch));
        A(dalloc(h, &x->r_final, c.max_batch));
        A(dalloc(h, &x->r_touchoff, c.max_batch));
        A(dalloc(h, &x->info, 1));
    }
    if (e != cudaSuccess) {
        dm_destroy(h);
        return e == cudaErrorMemoryAllocation ? DM_ERR_OOM : DM_ERR_CUDA;
    }
    h->dh.ad_step = 0;   // dm_hash_prompts hashes the fixed length
    h->dh.Kf2 = c.route_prefix_blocks;
    for (uint32_t f = 0; f < d.nrings; ++f) {
        d.ring[f].vpos = h->vpos_buf[f][0];
        d.ring[f].owner = h->owner_buf[f][0];
        d.ring[f].vidx = h->vidx_buf[f][0];
        h->dh.ring[f] = d.ring[f];
    }
    set_levels(d, 0);
    A(cudaMemcpyAsync(kx_dev, kx, sizeof(kx), cudaMemcpyHostToDevice, h->st));
    A(cudaMemsetAsync(d.seg_pub, 0, d.max_segs * sizeof(dm::SegPub), h->st));
    A(cudaMemsetAsync(d.inst_state, 0, M, h->st));
    A(cudaMemsetAsync(d.W, 0, M * 8, h->st));
    if (d.KQ) {
        A(cudaMemsetAsync(d.kr_head, 0, M * 8, h->st));
        A(cudaMemsetAsync(d.kr_tail, 0, M * 8, h->st));
        A(cudaMemsetAsync(d.kring, 0, M * d.KQ * 8, h->st));
    }
    A(cudaMemsetAsync(d.metrics, 0, sizeof(dm::DevMetrics), h->st));
    if (c.adapt_step_blocks) {
        A(cudaMemsetAsync(d.ad_set, 0, (d.ad_set_mask + 1) * 8, h->st));
        A(cudaMemsetAsync(d.ad_cnt, 0, (d.ad_cnt_mask + 1) * sizeof(dm::AdCount), h->st));
    }
    A(cudaMemsetAsync(d.q_head, 0, M * 4, h->st));
    A(cudaMemsetAsync(d.q_tail, 0, M * 4, h->st));
    A(cudaMemsetAsync(d.table, 0, M * 8, h->st));
    A(cudaMemsetAsync(d.logbuf, 0, M * 8, h->st));
    A(cudaMemsetAsync(d.table_alt, 0, M * 8, h->st));
    A(cudaMemsetAsync(d.pool, 0, uint64_t(h->pool_target) * 8, h->st));
    A(cudaMemsetAsync(d.rb_rr, 0, 4, h->st));
    A(cudaMemsetAsync(d.logbuf_alt, 0, M * 8, h->st));
    A(cudaMemsetAsync(d.stale, 0, M * 8, h->st));
    A(cudaMemsetAsync(d.stale_alt, 0, M * 8, h->st));
    A(cudaMemsetAsync(d.loghome, 0, M * 8, h->st));
    A(cudaMemsetAsync(d.loghome_alt, 0, M * 8, h->st));
    A(cudaMemsetAsync(d.mt_flags, 0, M * 4, h->st));
    A(cudaMemsetAsync(d.log_front, 0, M * 8, h->st));
    A(cudaMemsetAsync(d.log_tail, 0, M * 8, h->st));
    A(cudaMemsetAsync(d.live, 0, M * 8, h->st));
    A(cudaMemsetAsync(d.used, 0, M * 8, h->st));
    A(cudaMemsetAsync(d.clock, 0, 8, h->st));
    A(cudaMemsetAsync(d.maint_count, 0, 16, h->st));
    A(cudaMemsetAsync(d.err, 0, 4, h->st));
    A(cudaMemsetAsync(h->d.info, 0, sizeof(dm::BatchInfo), h->st));
    A(cudaMemsetAsync(h->dh.info, 0, sizeof(dm::BatchInfo), h->st));
    A(dm::launch_next_live(d, h->st));
    A(cudaStreamSynchronize(h->st));
    if (e != cudaSuccess) {
        dm_destroy(h);
        return DM_ERR_CUDA;
    }
    h->state.assign(M, 0);
    h->tables.assign(M, nullptr);
    h->logs.assign(M, nullptr);

    h->logs2.assign(M, nullptr);
    h->stales.assign(M, nullptr);
    h->stales2.assign(M, nullptr);
    h->homes.assign(M, nullptr);
    h->homes2.assign(M, nullptr);
    h->hash_grid = dm::hash_grid_size();
    *out = h;
    return DM_OK;
}

// Keep the hash-prompts copy in step with the ring / instance state.
static void sync_copy(dm_handle *h) {
    DevState keep = h->dh;
    h->dh = h->d;
    h->dh.r_L = keep.r_L; h->dh.r_nblk = keep.r_nblk; h->dh.r_segoff = keep.r_segoff;
    h->dh.r_tokoff = keep.r_tokoff; h->dh.r_blkoff = keep.r_blkoff; h->dh.seg_req = keep.seg_req;
    h->dh.seg_total = keep.seg_total; h->dh.seg_carry = keep.seg_carry; h->dh.plocal = keep.plocal;
    h->dh.seg_total2 = keep.seg_total2;
    h->dh.r_c1 = keep.r_c1; h->dh.r_c2 = keep.r_c2;
    h->dh.r_final = keep.r_final; h->dh.r_touchoff = keep.r_touchoff;
    h->dh.info = keep.info;
}

static dm_status ring_change(dm_handle *h, uint32_t id, bool add) {
    DevState &d = h->d;
    const uint32_t newR = add ? d.R + d.V : d.R - d.V;
    uint64_t *nv[dm::kMaxD] = {};
    uint32_t *no[dm::kMaxD] = {}, *ni[dm::kMaxD] = {};
    for (uint32_t f = 0; f < d.nrings; ++f) {
        const int nb = 1 - h->cur[f];
        nv[f] = h->vpos_buf[f][nb];
        no[f] = h->owner_buf[f][nb];
        ni[f] = h->vidx_buf[f][nb];
    }
    cudaError_t e = dm::launch_ring_update(d, id, add, h->ring_spos, h->ring_svidx, nv, no, ni, h->st);
    if (e != cudaSuccess) return map_cuda(h, e);
    for (uint32_t f = 0; f < d.nrings; ++f) {
        h->cur[f] = 1 - h->cur[f];
        d.ring[f].vpos = nv[f];
        d.ring[f].owner = no[f];
        d.ring[f].vidx = ni[f];
    }
    set_levels(d, newR);
    e = dm::launch_tree_build(d, h->st);
    if (e == cudaSuccess) e = dm::launch_set_state(d, id, add ? 1 : 2, h->st);
    if (e == cudaSuccess) e = dm::launch_next_live(d, h->st);
    sync_copy(h);
    return map_cuda(h, e);
}

dm_status dm_add_instance(dm_handle *h, uint32_t id) {
    dm_status s = check_live(h);
    if (s) return s;
    if (h->shard_open) return DM_ERR_ORDER;   // a sharded batch is between begin and finish
    DevState &d = h->d;
    if (id >= d.M) return DM_ERR_INVALID_ARG;
    if (h->state[id] == 1) return DM_ERR_DUPLICATE_ID;
    cudaError_t e = cudaSuccess;
    if (h->state[id] == 2) {
        uint32_t ht[2];
        e = cudaMemcpyAsync(&ht[0], d.q_head + id, 4, cudaMemcpyDeviceToHost, h->st);
        if (e == cudaSuccess) e = cudaMemcpyAsync(&ht[1], d.q_tail + id, 4, cudaMemcpyDeviceToHost, h->st);
        if (e == cudaSuccess) e = cudaStreamSynchronize(h->st);
        if (e != cudaSuccess) return map_cuda(h, e);
        if (ht[0] != ht[1]) return DM_ERR_DUPLICATE_ID;
    }
    Slot *cur = h->tables[id];   // the index this id uses now (rebuilds trade buffers with the pool)
    const bool first = cur == nullptr;
    if (first) {
        Slot *t = nullptr, *spare = nullptr;
        Rec *lg = nullptr, *lg2 = nullptr;
        uint8_t *sf = nullptr, *sf2 = nullptr;
        uint32_t *hm = nullptr, *hm2 = nullptr;
        e = dalloc(h, &t, d.S);
        if (e == cudaSuccess && d.pool_n < h->pool_target) e = dalloc(h, &spare, d.S);
        if (e == cudaSuccess) e = dalloc(h, &lg, d.logcap);
        if (e == cudaSuccess) e = dalloc(h, &lg2, d.logcap);
        if (e == cudaSuccess) e = dalloc(h, &sf, d.logcap);
        if (e == cudaSuccess) e = dalloc(h, &sf2, d.logcap);
        if (e == cudaSuccess) e = dalloc(h, &hm, d.logcap);
        if (e == cudaSuccess) e = dalloc(h, &hm2, d.logcap);
        if (e != cudaSuccess) { cudaGetLastError(); return DM_ERR_OOM; }
        if (spare) {
            e = cudaMemcpyAsync(d.pool + d.pool_n, &spare, sizeof(Slot *), cudaMemcpyHostToDevice, h->st);
            if (e == cudaSuccess) e = cudaStreamSynchronize(h->st);
            if (e != cudaSuccess) return map_cuda(h, e);
            ++h->d.pool_n;
        }
        h->tables[id] = t;
        cur = t;
        h->logs[id] = lg;
        h->logs2[id] = lg2;
        h->stales[id] = sf;
        h->stales2[id] = sf2;
        h->homes[id] = hm;
        h->homes2[id] = hm2;
    }
    if (!first) {   // a re-added id keeps whichever index buffer it holds now
        e = cudaMemcpyAsync(&cur, d.table + id, sizeof(Slot *), cudaMemcpyDeviceToHost, h->st);
        if (e == cudaSuccess) e = cudaStreamSynchronize(h->st);
        if (e != cudaSuccess) return map_cuda(h, e);
    }
    // a (re-)added instance starts empty, both buffers of each log
    struct { void *dst; const void *src; } ptrs[] = {
        {d.table + id, &cur},
        {d.logbuf + id, &h->logs[id]}, {d.logbuf_alt + id, &h->logs2[id]},
        {d.stale + id, &h->stales[id]}, {d.stale_alt + id, &h->stales2[id]},
        {d.loghome + id, &h->homes[id]}, {d.loghome_alt + id, &h->homes2[id]}};
    for (auto &pp : ptrs)
        if (e == cudaSuccess) e = cudaMemcpyAsync(pp.dst, pp.src, sizeof(void *), cudaMemcpyHostToDevice, h->st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(h->st);
    if (e != cudaSuccess) return map_cuda(h, e);
    e = cudaMemsetAsync(cur, 0, d.S * sizeof(Slot), h->st);
    if (e == cudaSuccess) e = cudaMemsetAsync(h->stales[id], 0, d.logcap, h->st);
    if (e == cudaSuccess) e = cudaMemsetAsync(h->stales2[id], 0, d.logcap, h->st);
    if (e == cudaSuccess) e = cudaMemsetAsync(d.log_front + id, 0, 8, h->st);
    if (e == cudaSuccess) e = cudaMemsetAsync(d.log_tail + id, 0, 8, h->st);
    if (e == cudaSuccess) e = cudaMemsetAsync(d.live + id, 0, 8, h->st);
    if (e == cudaSuccess) e = cudaMemsetAsync(d.used + id, 0, 8, h->st);
    if (e == cudaSuccess) e = cudaMemsetAsync(d.W + id, 0, 8, h->st);
    if (e == cudaSuccess) e = cudaMemsetAsync(d.q_head + id, 0, 4, h->st);
    if (e == cudaSuccess) e = cudaMemsetAsync(d.q_tail + id, 0, 4, h->st);
    if (e != cudaSuccess) return map_cuda(h, e);
    s = ring_change(h, id, true);
    if (s) return s;
    h->state[id] = 1;
    h->n_live++;
    return DM_OK;
}

dm_status dm_remove_instance(dm_handle *h, uint32_t id) {
    dm_status s = check_live(h);
    if (s) return s;
    if (h->shard_open) return DM_ERR_ORDER;   // a sharded batch is between begin and finish
    if (id >= h->d.M || h->state[id] != 1) return DM_ERR_UNKNOWN_ID;
    s = ring_change(h, id, false);
    if (s) return s;
    h->state[id] = 2;
    h->n_live--;
    return DM_OK;
}

static dm_status check_batch(dm_handle *h, const dm_batch *b, const dm_route_out *o) {
    dm_status s = check_live(h);
    if (s) return s;
    if (!b || b->reserved0) return DM_ERR_INVALID_ARG;
    if (b->n > 0 && (!b->tokens || !b->offsets || !b->lengths)) return DM_ERR_INVALID_ARG;
    if (o && b->n > 0 &&
        (!o->cand1 || !o->cand2 || !o->hit1 || !o->hit2 || !o->ttft1 || !o->ttft2 || !o->chosen || !o->switched))
        return DM_ERR_INVALID_ARG;
    if (b->n > h->d.max_batch || b->total_tokens > h->cfg.max_batch_tokens) return DM_ERR_CAPACITY;
    return DM_OK;
}

// The hashing kernel reads prompts with 16-byte loads.
static bool tokens_aligned(const dm_batch *b) {
    return b->n == 0 || (reinterpret_cast<uintptr_t>(b->tokens) & 15) == 0;
}

// A handle made for d candidates (dm_config.candidates not 0 or 2) routes only
// through dm_route_batch_d and does not rebalance.
static bool pair_handle(const dm_handle *h) { return h->cfg.candidates == 0 || h->cfg.candidates == 2; }

// Routing, first half: time, drain and layout, then the routing kernel for
// requests r0 .. r1-1 (all of them, or one shard).
static dm_status route_begin(dm_handle *h, const dm_batch *b, uint32_t r0, uint32_t r1) {
    if (!pair_handle(h)) return DM_ERR_INVALID_ARG;
    if (!tokens_aligned(b)) return DM_ERR_INVALID_ARG;
    if (h->n_live < 2) return DM_ERR_NO_INSTANCES;
    if (h->have_time && b->batch_time_us < h->t_prev) return DM_ERR_ORDER;
    const uint64_t delta = h->have_time ? b->batch_time_us - h->t_prev : 0;
    const uint64_t t0 = h->have_time ? h->t_prev : b->batch_time_us;   // start of the drain window
    h->t_prev = b->batch_time_us;
    h->have_time = true;
    h->pending = false;   // the batch scratch now holds this batch
    const DevState &d = h->d;
    cudaError_t e;
    { Stage st(h, DM_STAGE_SETUP); e = dm::launch_setup_route(d, *b, delta, t0, h->st); }   // drain included
    if (e == cudaSuccess && b->n) {   // hashing, ring lookup and probes: one kernel
        Stage st(h, DM_STAGE_HASH);
        // a fresh epoch mask per call: records of earlier batches never pass its check
        const uint64_t E = dm::fmix64(++h->epoch ^ 0x6a09e667f3bcc909ull);
        e = dm::launch_hash_probe(d, *b, E, r0, r1, h->st);
    }
    return e == cudaSuccess ? DM_OK : map_cuda(h, e);
}

// Routing, second half: carries, choices in arrival order, queues,
// metrics, the adaptive window; the batch becomes the pending commit.
static dm_status route_finish(dm_handle *h, const dm_batch *b, const dm_route_out *o) {
    const DevState &d = h->d;
    cudaError_t e = cudaSuccess;
    if (b->n) {
        Stage st(h, DM_STAGE_CHOICE);
        e = dm::launch_choice(d, *o, b->n, h->seq_next, b->batch_time_us, h->st);
    }
    if (e == cudaSuccess && b->n && d.ad_step) {
        // end of an adaptive window: rebuild the expanded nodes into the
        // other table, restart the counts; the next batch walks the new tree
        h->ad_T += b->n;
        if (++h->ad_batches == h->cfg.adapt_window) {
            e = cudaMemsetAsync(h->ad_alt, 0, (d.ad_set_mask + 1) * 8, h->st);
            if (e == cudaSuccess) e = dm::launch_adapt_update(d, h->ad_alt, h->n_live, h->ad_T, h->st);
            if (e == cudaSuccess)
                e = cudaMemsetAsync(d.ad_cnt, 0, (d.ad_cnt_mask + 1) * sizeof(dm::AdCount), h->st);
            std::swap(h->d.ad_set, h->ad_alt);
            h->ad_T = 0;
            h->ad_batches = 0;
        }
    }
    if (e != cudaSuccess) return map_cuda(h, e);
    h->pending = true;
    h->pending_n = b->n;
    h->pending_seq0 = h->seq_next;
    h->seq_next += b->n;
    return DM_OK;
}

dm_status dm_route_batch(dm_handle *h, const dm_batch *b, const dm_route_out *o) {
    dm_status s = check_batch(h, b, o);
    if (s) return s;
    if (!o) return DM_ERR_INVALID_ARG;
    if (h->shard_open) return DM_ERR_ORDER;
    s = route_begin(h, b, 0, b->n);
    return s ? s : route_finish(h, b, o);
}

dm_status dm_route_shard_begin(dm_handle *h, const dm_batch *b, uint32_t r0, uint32_t r1) {
    dm_status s = check_batch(h, b, nullptr);
    if (s) return s;
    if (r0 > r1 || r1 > b->n || h->d.ad_step) return DM_ERR_INVALID_ARG;
    if (h->shard_open) return DM_ERR_ORDER;
    s = route_begin(h, b, r0, r1);
    if (s) return s;
    h->shard_open = true;
    h->shard_n = b->n;
    return DM_OK;
}

dm_status dm_shard_export(dm_handle *h, uint32_t r0, uint32_t r1, void *buf_dev, uint64_t cap, uint64_t *bytes_dev) {
    dm_status s = check_live(h);
    if (s) return s;
    if (!h->shard_open || r0 > r1 || r1 > h->shard_n || (r1 > r0 && !buf_dev)) return DM_ERR_INVALID_ARG;
    const cudaError_t e = dm::launch_shard_copy(h->d, true, r0, r1, static_cast<uint8_t *>(buf_dev), cap,
                                                static_cast<uint64_t *>(bytes_dev), h->st);
    return e == cudaSuccess ? DM_OK : map_cuda(h, e);
}

dm_status dm_shard_import(dm_handle *h, uint32_t r0, uint32_t r1, const void *buf_dev, uint64_t bytes) {
    dm_status s = check_live(h);
    if (s) return s;
    if (!h->shard_open || r0 > r1 || r1 > h->shard_n || (r1 > r0 && !buf_dev)) return DM_ERR_INVALID_ARG;
    const cudaError_t e = dm::launch_shard_copy(h->d, false, r0, r1,
                                                static_cast<uint8_t *>(const_cast<void *>(buf_dev)), bytes, nullptr,
                                                h->st);
    return e == cudaSuccess ? DM_OK : map_cuda(h, e);
}

dm_status dm_route_shard_finish(dm_handle *h, const dm_batch *b, const dm_route_out *o) {
    dm_status s = check_batch(h, b, o);
    if (s) return s;
    if (!o || !h->shard_open || b->n != h->shard_n) return DM_ERR_INVALID_ARG;
    h->shard_open = false;
    return route_finish(h, b, o);
}

dm_status dm_route_batch_host_async(dm_handle *h, const dm_batch *b, const dm_route_out *o) {
    dm_status s = check_batch(h, b, o);
    if (s) return s;
    if (h->shard_open) return DM_ERR_ORDER;   // a sharded batch is between begin and finish
    if (!pair_handle(h)) return DM_ERR_INVALID_ARG;
    if (!o) return DM_ERR_INVALID_ARG;
    cudaError_t e = cudaSuccess;
    const uint32_t mb = h->d.max_batch;
    if (!h->copy_st) {
        auto A = [&](cudaError_t x) { if (e == cudaSuccess) e = x; };
        for (auto &x : h->hs) {
            A(dalloc(h, &x.tokens, h->cfg.max_batch_tokens + 4));
            A(dalloc(h, &x.offsets, mb));
            A(dalloc(h, &x.lengths, mb));
            A(dalloc(h, &x.out.cand1, mb));
            A(dalloc(h, &x.out.cand2, mb));
            A(dalloc(h, &x.out.hit1, mb));
            A(dalloc(h, &x.out.hit2, mb));
            A(dalloc(h, &x.out.ttft1, mb));
            A(dalloc(h, &x.out.ttft2, mb));
            A(dalloc(h, &x.out.chosen, mb));
            A(dalloc(h, &x.out.switched, mb));
            A(cudaEventCreateWithFlags(&x.copied, cudaEventDisableTiming));
            A(cudaEventCreateWithFlags(&x.consumed, cudaEventDisableTiming));
        }
        A(cudaStreamCreateWithFlags(&h->copy_st, cudaStreamNonBlocking));
        if (e != cudaSuccess) { cudaGetLastError(); h->copy_st = nullptr; return DM_ERR_OOM; }
    }
    auto &x = h->hs[h->hs_next];
    h->hs_next ^= 1;
    const uint32_t n = b->n;
    if (n) {
        // the upload waits until kernels reading this buffer's last batch are done
        if (x.used) e = cudaStreamWaitEvent(h->copy_st, x.consumed, 0);
        if (e == cudaSuccess)
            e = cudaMemcpyAsync(x.tokens, b->tokens, b->total_tokens * 4, cudaMemcpyHostToDevice, h->copy_st);
        if (e == cudaSuccess) e = cudaMemcpyAsync(x.offsets, b->offsets, n * 8ull, cudaMemcpyHostToDevice, h->copy_st);
        if (e == cudaSuccess) e = cudaMemcpyAsync(x.lengths, b->lengths, n * 4ull, cudaMemcpyHostToDevice, h->copy_st);
        if (e == cudaSuccess) e = cudaEventRecord(x.copied, h->copy_st);
        if (e == cudaSuccess) e = cudaStreamWaitEvent(h->st, x.copied, 0);
        if (e != cudaSuccess) return map_cuda(h, e);
    }
    dm_batch db = *b;
    db.tokens = x.tokens;
    db.offsets = x.offsets;
    db.lengths = x.lengths;
    s = dm_route_batch(h, &db, &x.out);
    if (s) return s;
    if (n) {
        e = cudaEventRecord(x.consumed, h->st);
        x.used = true;
        struct { void *dst; const void *src; size_t bytes; } cp[] = {
            {o->cand1, x.out.cand1, n * 4ull}, {o->cand2, x.out.cand2, n * 4ull}, {o->hit1, x.out.hit1, n * 4ull},
            {o->hit2, x.out.hit2, n * 4ull}, {o->ttft1, x.out.ttft1, n * 8ull}, {o->ttft2, x.out.ttft2, n * 8ull},
            {o->chosen, x.out.chosen, n * 4ull}, {o->switched, x.out.switched, n * 1ull}};
        for (auto &c : cp)
            if (e == cudaSuccess) e = cudaMemcpyAsync(c.dst, c.src, c.bytes, cudaMemcpyDeviceToHost, h->st);
    }
    return map_cuda(h, e);
}

dm_status dm_route_batch_d(dm_handle *h, const dm_batch *b, const dm_route_out_d *o) {
    dm_status s = check_batch(h, b, nullptr);
    if (s) return s;
    if (h->shard_open) return DM_ERR_ORDER;   // a sharded batch is between begin and finish
    if (!tokens_aligned(b) || !o) return DM_ERR_INVALID_ARG;
    if (b->n > 0 && (!o->cand || !o->hit || !o->ttft || !o->chosen || !o->switched)) return DM_ERR_INVALID_ARG;
    const DevState &d = h->d;
    if (h->n_live < 2 || h->n_live < d.nd) return DM_ERR_NO_INSTANCES;
    if (h->have_time && b->batch_time_us < h->t_prev) return DM_ERR_ORDER;
    const uint64_t delta = h->have_time ? b->batch_time_us - h->t_prev : 0;
    const uint64_t t0 = h->have_time ? h->t_prev : b->batch_time_us;
    h->t_prev = b->batch_time_us;
    h->have_time = true;
    cudaError_t e;
    { Stage st(h, DM_STAGE_SETUP); e = dm::launch_setup_plain_drain(d, *b, delta, t0, h->st); }
    if (e == cudaSuccess && b->n) { Stage st(h, DM_STAGE_HASH); e = dm::launch_hash(d, *b, h->hash_grid, h->st); }
    if (e == cudaSuccess && b->n) {
        Stage st(h, DM_STAGE_CHOICE);   // ring lookups, probes and the choice
        e = dm::launch_route_d(d, *b, *o, h->seq_next, h->st);
    }
    if (e != cudaSuccess) return map_cuda(h, e);
    h->pending = true;
    h->pending_n = b->n;
    h->pending_seq0 = h->seq_next;
    h->seq_next += b->n;
    return DM_OK;
}

dm_status dm_route_batch_host(dm_handle *h, const dm_batch *b, const dm_route_out *o) {
    dm_status s = dm_route_batch_host_async(h, b, o);
    if (s) return s;
    return map_cuda(h, cudaStreamSynchronize(h->st));
}

dm_status dm_rebalance(dm_handle *h, dm_migration *out_host, uint32_t cap, uint32_t *n_out) {
    dm_status s = check_live(h);
    if (s) return s;
    if (h->shard_open) return DM_ERR_ORDER;   // a sharded batch is between begin and finish
    if (!pair_handle(h)) return DM_ERR_INVALID_ARG;
    if (!n_out || (cap && !out_host)) return DM_ERR_INVALID_ARG;
    if (cap > h->rb_out_cap || !h->rb_n_dev) {   // device staging of the results
        dm_migration *buf = nullptr;
        uint32_t *cnt = h->rb_n_dev;
        cudaError_t e = dalloc(h, &buf, cap ? cap : 1);
        if (e == cudaSuccess && !cnt) e = dalloc(h, &cnt, 1);
        if (e != cudaSuccess) { cudaGetLastError(); return DM_ERR_OOM; }
        h->rb_out_dev = buf;
        h->rb_out_cap = cap ? cap : 1;
        h->rb_n_dev = cnt;
    }
    s = dm_rebalance_async(h, h->rb_out_dev, cap, h->rb_n_dev);
    if (s) return s;
    uint32_t n = 0;
    cudaError_t e = cudaMemcpyAsync(&n, h->rb_n_dev, 4, cudaMemcpyDeviceToHost, h->st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(h->st);
    if (e == cudaSuccess && n && cap)
        e = cudaMemcpy(out_host, h->rb_out_dev, sizeof(dm_migration) * (n < cap ? n : cap), cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) return map_cuda(h, e);
    *n_out = n;
    return DM_OK;
}

dm_status dm_rebalance_async(dm_handle *h, dm_migration *out_dev, uint32_t cap, uint32_t *n_out_dev) {
    dm_status s = check_live(h);
    if (s) return s;
    if (h->shard_open) return DM_ERR_ORDER;   // a sharded batch is between begin and finish
    if (!pair_handle(h)) return DM_ERR_INVALID_ARG;
    if (!n_out_dev || (cap && !out_dev)) return DM_ERR_INVALID_ARG;
    const uint32_t n = h->pending ? h->pending_n : 0;
    cudaError_t e;
    {
        Stage st(h, DM_STAGE_REBALANCE);
        e = dm::launch_rebalance(h->d, n, h->pending_seq0, ++h->rebalance_calls, out_dev, cap, n_out_dev, h->st);
    }
    return map_cuda(h, e);
}

dm_status dm_commit_cache(dm_handle *h) {
    dm_status s = check_live(h);
    if (s) return s;
    if (h->shard_open) return DM_ERR_ORDER;   // a sharded batch is between begin and finish
    if (!h->pending) return DM_OK;
    cudaError_t e;
    {
        Stage st(h, DM_STAGE_COMMIT);
        e = dm::launch_commit(h->d, h->pending_n, h->st);
    }
    h->pending = false;
    return map_cuda(h, e);
}

dm_status dm_hash_prompts(dm_handle *h, const dm_batch *b, uint64_t *keys_dev, uint64_t *key_off_dev,
                          uint64_t *pos_dev) {
    dm_status s = check_batch(h, b, nullptr);
    if (s) return s;
    if (h->shard_open) return DM_ERR_ORDER;   // a sharded batch is between begin and finish
    if (b->n && (!keys_dev || !key_off_dev || !pos_dev)) return DM_ERR_INVALID_ARG;
    if (!tokens_aligned(b)) return DM_ERR_INVALID_ARG;
    if (b->n == 0) return DM_OK;
    cudaError_t e = dm::launch_setup(h->dh, *b, h->st);
    if (e == cudaSuccess) e = dm::launch_hash(h->dh, *b, h->hash_grid, h->st);
    if (e == cudaSuccess) e = dm::launch_hash_keys(h->dh, b->n, keys_dev, key_off_dev, pos_dev, h->st);
    return map_cuda(h, e);
}

dm_status dm_ring_lookup(dm_handle *h, const uint64_t *pos_dev, uint32_t n, uint32_t *o1, uint32_t *o2) {
    dm_status s = check_live(h);
    if (s) return s;
    if (n && (!pos_dev || !o1 || !o2)) return DM_ERR_INVALID_ARG;
    if (n && h->d.R == 0) return DM_ERR_NO_INSTANCES;
    return map_cuda(h, dm::launch_ring_lookup(h->d, pos_dev, n, o1, o2, h->st));
}

dm_status dm_get_loads(dm_handle *h, uint64_t *W_host, uint32_t cap, uint32_t *n_out) {
    dm_status s = check_handle(h);
    if (s) return s;
    if (!n_out || (!W_host && cap)) return DM_ERR_INVALID_ARG;
    const uint32_t k = cap < h->d.M ? cap : h->d.M;
    cudaError_t e = k ? cudaMemcpyAsync(W_host, h->d.W, k * 8ull, cudaMemcpyDeviceToHost, h->st) : cudaSuccess;
    if (e == cudaSuccess) e = cudaStreamSynchronize(h->st);
    if (e != cudaSuccess) return map_cuda(h, e);
    *n_out = h->d.M;
    return DM_OK;
}

dm_status dm_export_cache(dm_handle *h, uint32_t id, uint64_t *keys, uint64_t *stamps, uint64_t cap,
                          uint64_t *n_out) {
    dm_status s = check_handle(h);
    if (s) return s;
    if (id >= h->d.M || !n_out || (cap && (!keys || !stamps))) return DM_ERR_INVALID_ARG;
    *n_out = 0;
    if (!h->tables[id]) return DM_OK;
    Slot *cur = nullptr;   // the buffers in use (rebuilds and compactions swap them)
    Rec *lcur = nullptr;
    uint64_t front = 0;
    cudaError_t e = cudaMemcpyAsync(&cur, h->d.table + id, sizeof(Slot *), cudaMemcpyDeviceToHost, h->st);
    if (e == cudaSuccess) e = cudaMemcpyAsync(&lcur, h->d.logbuf + id, sizeof(Rec *), cudaMemcpyDeviceToHost, h->st);
    if (e == cudaSuccess) e = cudaMemcpyAsync(&front, h->d.log_front + id, 8, cudaMemcpyDeviceToHost, h->st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(h->st);
    if (e != cudaSuccess) return map_cuda(h, e);
    std::vector<Slot> t(h->d.S);
    std::vector<Rec> lg(h->d.logcap);
    e = cudaMemcpyAsync(t.data(), cur, h->d.S * sizeof(Slot), cudaMemcpyDeviceToHost, h->st);
    if (e == cudaSuccess)
        e = cudaMemcpyAsync(lg.data(), lcur, h->d.logcap * sizeof(Rec), cudaMemcpyDeviceToHost, h->st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(h->st);
    if (e != cudaSuccess) return map_cuda(h, e);
    uint64_t k = 0;
    for (const Slot &x : t) {
        if (x.key == 0 || x.pos1 == 0 || x.pos1 - 1 < front) continue;   // empty or evicted
        if (k < cap) {
            keys[k] = x.key;
            stamps[k] = lg[(x.pos1 - 1) & (h->d.logcap - 1)].stamp;
        }
        ++k;
    }
    *n_out = k;
    return DM_OK;
}

dm_status dm_export_queue(dm_handle *h, uint32_t id, uint64_t *seq, uint64_t *work, uint64_t *rem, uint64_t cap,
                          uint64_t *n_out) {
    dm_status s = check_handle(h);
    if (s) return s;
    if (id >= h->d.M || !n_out || (cap && (!seq || !work || !rem))) return DM_ERR_INVALID_ARG;
    uint32_t ht[2];
    std::vector<QEntry> q(h->d.Q);
    cudaError_t e = cudaMemcpyAsync(&ht[0], h->d.q_head + id, 4, cudaMemcpyDeviceToHost, h->st);
    if (e == cudaSuccess) e = cudaMemcpyAsync(&ht[1], h->d.q_tail + id, 4, cudaMemcpyDeviceToHost, h->st);
    if (e == cudaSuccess)
        e = cudaMemcpyAsync(q.data(), h->d.q + uint64_t(id) * h->d.Q, h->d.Q * sizeof(QEntry),
                            cudaMemcpyDeviceToHost, h->st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(h->st);
    if (e != cudaSuccess) return map_cuda(h, e);
    uint64_t k = 0;
    for (uint32_t p = ht[0]; p != ht[1]; ++p) {
        const QEntry &x = q[p & (h->d.Q - 1)];
        if (x.moved == dm::kTomb) continue;
        if (k < cap) { seq[k] = x.seq; work[k] = x.work; rem[k] = x.remaining; }
        ++k;
    }
    *n_out = k;
    return DM_OK;
}

dm_status dm_export_ring(dm_handle *h, int f, uint64_t *vpos, uint32_t *owner, uint32_t cap, uint32_t *n_out) {
    dm_status s = check_handle(h);
    if (s) return s;
    if (f < 0 || (uint32_t)f >= h->d.nrings || !n_out || (cap && (!vpos || !owner))) return DM_ERR_INVALID_ARG;
    const uint32_t k = cap < h->d.R ? cap : h->d.R;
    cudaError_t e = cudaMemcpyAsync(vpos, h->d.ring[f].vpos, k * 8ull, cudaMemcpyDeviceToHost, h->st);
    if (e == cudaSuccess) e = cudaMemcpyAsync(owner, h->d.ring[f].owner, k * 4ull, cudaMemcpyDeviceToHost, h->st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(h->st);
    *n_out = h->d.R;
    return map_cuda(h, e);
}

dm_status dm_get_clock(dm_handle *h, uint64_t *clock_host) {
    dm_status s = check_handle(h);
    if (s) return s;
    if (!clock_host) return DM_ERR_INVALID_ARG;
    cudaError_t e = cudaMemcpyAsync(clock_host, h->d.clock, 8, cudaMemcpyDeviceToHost, h->st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(h->st);
    return map_cuda(h, e);
}

dm_status dm_get_maint_counts(dm_handle *h, uint64_t *rebuilds_host, uint64_t *compactions_host) {
    dm_status s = check_handle(h);
    if (s) return s;
    if (!rebuilds_host || !compactions_host) return DM_ERR_INVALID_ARG;
    uint64_t c[2] = {0, 0};
    cudaError_t e = cudaMemcpyAsync(c, h->d.maint_count, 16, cudaMemcpyDeviceToHost, h->st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(h->st);
    if (e != cudaSuccess) return map_cuda(h, e);
    *rebuilds_host = c[0];
    *compactions_host = c[1];
    return DM_OK;
}

dm_status dm_get_route_blocks(dm_handle *h, uint32_t *out_dev, uint32_t n) {
    dm_status s = check_handle(h);
    if (s) return s;
    if (n > h->pending_n || (n && !out_dev)) return DM_ERR_INVALID_ARG;
    if (n == 0) return DM_OK;
    cudaError_t e = cudaMemcpyAsync(out_dev, h->d.r_K, n * sizeof(uint32_t), cudaMemcpyDeviceToDevice, h->st);
    return e == cudaSuccess ? DM_OK : map_cuda(h, e);
}

dm_status dm_export_prefix_tree(dm_handle *h, uint64_t *keys_host, uint64_t cap, uint64_t *n_out) {
    dm_status s = check_handle(h);
    if (s) return s;
    if (!n_out || (cap && !keys_host)) return DM_ERR_INVALID_ARG;
    *n_out = 0;
    if (!h->d.ad_step) return DM_OK;
    std::vector<uint64_t> t(h->d.ad_set_mask + 1);
    cudaError_t e = cudaMemcpyAsync(t.data(), h->d.ad_set, t.size() * 8, cudaMemcpyDeviceToHost, h->st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(h->st);
    if (e != cudaSuccess) return map_cuda(h, e);
    uint64_t k = 0;
    for (uint64_t x : t)
        if (x) {
            if (k < cap) keys_host[k] = x;
            ++k;
        }
    *n_out = k;
    return DM_OK;
}

// Lower edge of the histogram bucket holding the ceil(pnum/pden * count)-th
// smallest value (0 for an empty histogram).
static uint64_t hist_quantile(const unsigned long long *hist, uint64_t count, uint64_t pnum, uint64_t pden) {
    if (count == 0) return 0;
    uint64_t rank = (pnum * count + pden - 1) / pden;
    if (rank == 0) rank = 1;
    uint64_t cum = 0;
    uint32_t k = 0;
    for (; k + 1 < dm::kHistBuckets; ++k) {
        cum += hist[k];
        if (cum >= rank) break;
    }
    if (k < 16) return k;
    const uint32_t e = 4 + (k - 16) / 16, sub = (k - 16) % 16;
    return uint64_t(16 + sub) << (e - 4);
}

dm_status dm_get_metrics(dm_handle *h, dm_metrics *out, uint64_t *hist_host, uint32_t hist_cap, int reset) {
    dm_status s = check_handle(h);
    if (s) return s;
    if (!out || (hist_cap && !hist_host)) return DM_ERR_INVALID_ARG;
    dm::DevMetrics m;
    cudaError_t e = cudaMemcpyAsync(&m, h->d.metrics, sizeof m, cudaMemcpyDeviceToHost, h->st);
    if (e == cudaSuccess && reset) e = cudaMemsetAsync(h->d.metrics, 0, sizeof m, h->st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(h->st);
    if (e != cudaSuccess) return map_cuda(h, e);
    dm::fold_cv(&m);   // the last batch's sample (the device folds it at the next batch)
    out->requests = m.requests;
    out->prompt_tokens = m.prompt_tokens;
    out->hit_tokens = m.hit_tokens;
    out->switched = m.switched;
    out->est_slo_met = m.est_slo_met;
    out->completed = m.completed;
    out->ttft_sum_us = m.ttft_sum;
    out->ttft_max_us = m.ttft_max;
    out->slo_met = m.slo_met;
    out->ttft_p50_us = hist_quantile(m.hist, m.completed, 50, 100);
    out->ttft_p90_us = hist_quantile(m.hist, m.completed, 90, 100);
    out->ttft_p99_us = hist_quantile(m.hist, m.completed, 99, 100);
    out->cv_samples = m.cv_samples;
    out->cv_sum = m.cv_sum;
    out->cv_last = m.cv_last;
    for (uint32_t k = 0; k < hist_cap && k < dm::kHistBuckets; ++k) hist_host[k] = m.hist[k];
    return DM_OK;
}

void dm_test_fail_alloc(int64_t n) {
    g_alloc_seq.store(0, std::memory_order_relaxed);
    g_fail_at.store(n, std::memory_order_relaxed);
}

dm_status dm_last_error(dm_handle *h) {
    if (!h) return DM_ERR_INVALID_ARG;
    if (h->sticky) return h->sticky;
    uint32_t err = 0;
    cudaError_t e = cudaMemcpyAsync(&err, h->d.err, 4, cudaMemcpyDeviceToHost, h->st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(h->st);
    if (e != cudaSuccess) return map_cuda(h, e);
    if (err) h->sticky = static_cast<dm_status>(err);
    return h->sticky;
}

dm_status dm_set_profiling(dm_handle *h, int on) {
    if (!h) return DM_ERR_INVALID_ARG;
    if (on == 0 || on == 1) {
        h->profiling = on ? (1u << DM_STAGE_COUNT) - 1u : 0u;
        return DM_OK;
    }
    if (!(on & DM_PROFILE_ONLY) || (on & ~(DM_PROFILE_ONLY | ((1 << DM_STAGE_COUNT) - 1)))) return DM_ERR_INVALID_ARG;
    h->profiling = (uint32_t)on & ((1u << DM_STAGE_COUNT) - 1u);
    return DM_OK;
}

dm_status dm_get_stage_times(dm_handle *h, double *ms, uint64_t *calls, int reset) {
    if (!h) return DM_ERR_INVALID_ARG;
    cudaError_t e = cudaStreamSynchronize(h->st);
    if (e != cudaSuccess) return map_cuda(h, e);
    for (auto &ev : h->events) {
        float t = 0.f;
        if (cudaEventElapsedTime(&t, ev.a, ev.b) == cudaSuccess) {
            h->stage_ms[ev.stage] += t;
            h->stage_calls[ev.stage] += 1;
        }
        h->ev_pool.push_back(ev.a);
        h->ev_pool.push_back(ev.b);
    }
    h->events.clear();
    for (int i = 0; i < DM_STAGE_COUNT; ++i) {
        if (ms) ms[i] = h->stage_ms[i];
        if (calls) calls[i] = h->stage_calls[i];
    }
    if (reset)
        for (int i = 0; i < DM_STAGE_COUNT; ++i) { h->stage_ms[i] = 0; h->stage_calls[i] = 0; }
    return DM_OK;
}

}  // extern "C"
