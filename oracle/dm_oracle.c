/*
 * dm_oracle.c -- plain, sequential CPU oracle of DualMap's per-batch routing
 * (arxiv 2602.06502).  TEST INFRASTRUCTURE ONLY: only the test-suite, the
 * smoke check and the benchmark's CPU-baseline leg may load this library.
 * It shares no code, header, table or constant generator with the CUDA path.
 *
 * Every step follows the paper's statement of the method, with the details
 * the paper leaves open fixed as listed below (the same readings the CUDA
 * path implements; each is argued in the design notes):
 *
 *   Hashing (Sec. 3.2 "two independent hash functions over the prompt
 *   prefix"; App. A.1.1 block-granular prefixes; App. A.3.2 per-block keys):
 *     key material from SplitMix64(seed), drawn in this order:
 *       K1[0..B) (low 32 bits of each draw), K2[0..B), G1|1, G2|1,
 *       S_c, S_r1, S_r2, S_v1, S_v2;
 *     block k of a prompt (tokens t_0..t_{B-1}) under function f:
 *       nh^f_k = sum_{i<B/2} ((t_2i + K^f_2i) mod 2^32)((t_2i+1 + K^f_2i+1) mod 2^32)  mod 2^64
 *       (the NH hash of Black et al., UMAC, CRYPTO 1999),
 *       d^f_k  = fmix64(nh^f_k + (k+1) G^f)        (MurmurHash3 finaliser),
 *       P^f_b  = sum_{k<=b} d^f_k  mod 2^64        (chained prefix value),
 *     cache key of block b: key_b = fmix64(P^1_b xor S_c), 0 replaced by 1;
 *     only full blocks are keyed (n_blk = floor(L/B));
 *     route positions: K = min(K_route, n_blk), pos_f = fmix64(P^f_{K-1} xor S_rf).
 *
 *   Dual rings (Sec. 3.4; App. A.1.3): each live id owns V virtual nodes per
 *     ring at vpos_f(id,v) = fmix64(mix64((id<<32)|v) xor S_vf), where mix64
 *     is one SplitMix64 output step; ring sorted by (vpos, id, v); a position
 *     p belongs to the first node with vpos >= p, wrapping to the first node
 *     (arcs (A,B] -> B).
 *
 *   Distinct candidates (Sec. 3.2, the unnumbered equation): c1 = owner on
 *     ring 1; c2 = owner on ring 2, or, if equal, the next live id after c1
 *     in ascending order, cyclically ((id1+1) mod N for dense ids).
 *
 *   Hit length (App. A.3.2): h_f = B * (leading run of keys resident on c_f),
 *     probed against the index as it was at the start of the batch.
 *
 *   TTFT and choice (Sec. 3.2 "SLO-aware strategy"; App. A.1.1 TTFT =
 *     T_q + T_c): ttft_f = W[c_f] + c*(L - h_f) in integer us, W = queued
 *     prefill work of the instance.  Equal hits: the less-loaded (by W, tie
 *     c1).  Otherwise the higher-hit candidate a unless ttft_a > SLO, then
 *     the less-loaded of the two (tie a), flagged "switched".  Loads update
 *     in arrival order within the batch; the request joins the chosen
 *     instance's FIFO queue with work c*(L - h_choice).
 *
 *   Choice rules.  Between the same two candidates (the ablation of Sec.
 *     4.3), with the rules of the compared schedulers (Sec. 2.2; Preble's
 *     and Mooncake's rules as the related-work appendix states them):
 *       DualMap         the SLO-aware rule above;
 *       cache affinity  the candidate with more hit tokens; equal hits: the
 *                       less-loaded by W, tie c1;
 *       least loaded    smaller W, tie c1 (hits ignored);
 *       min TTFT        smaller ttft_f = W[c_f] + c*(L - h_f), tie c1 (the
 *                       appendix prints it as a max of a difference; the
 *                       minimum of the sum is what the text describes);
 *       Preble          if the larger hit exceeds half the prompt
 *                       (2*max(h1,h2) > L): cache affinity, else min TTFT.
 *     For these, switched = 1 when the hits differ and the candidate with
 *     fewer of them was chosen.  Over all live instances (the baselines of
 *     Sec. 2.2 and Sec. 4), h_i probed on every live instance i:
 *       global cache affinity  c1, the owner on ring 1 (one prompt-aware
 *                              mapping, Sec. 1);
 *       global least loaded    smallest W_i, tie lowest id;
 *       global min TTFT        smallest W_i + c*(L - h_i), tie lowest id;
 *       global Preble          if 2*max_i h_i > L: among the instances with
 *                              that hit the smallest W_i, tie lowest id;
 *                              else global min TTFT;
 *     switched = 0; ttft1/ttft2 still report the two candidates; the queue
 *     entry's work is c*(L - h) of the chosen instance.
 *
 *   Time: batch time = arrival of the batch's last request; before routing,
 *     every instance's queue drains by the elapsed microseconds, starting
 *     at the previous batch time t0: an entry that finishes after w us of
 *     that window completes at t0 + w, and its TTFT is that minus the
 *     batch time it arrived with (kept when rebalancing moves it).
 *
 *   Metrics (Sec. 2.2 load-balance CV; Sec. 4.1 cache hit rate, SLO
 *     attainment, TTFT percentiles): per routed request its L, the hit
 *     tokens of the chosen candidate, switched, and whether the estimated
 *     TTFT on the chosen candidate is <= SLO; per completed entry its TTFT
 *     (sum, max, <= SLO count, and a log-linear histogram: values below 16
 *     exact, then 16 buckets per power of two); after the choices of a
 *     non-empty batch one CV sample over the live instances' W,
 *       CV = sqrt(n*S2 - S1^2) / S1,  S1 = sum W_i, S2 = sum W_i^2
 *     (the population CV of Sec. 2.2 with the n's cancelled; 0 when S1 = 0),
 *     with S1, S2 and n*S2 - S1^2 exact 128-bit integers, each turned into
 *     a double as double(hi)*2^64 + double(lo), every floating step rounded
 *     to nearest.
 *
 *   Commit (App. A.3.2 "KV cache save"): after route (and rebalance), in
 *     arrival order, each request touches its keys on its final instance,
 *     block n_blk-1 down to 0, each with stamp ++clock; an exact LRU of
 *     capacity C per instance.
 *
 *   Rebalance (Sec. 3.3, Eq. "rebalance"; App. A.1.2): hotspots are live
 *     instances with hot_den*N*W_i > hot_num*sum(W), taken in descending W;
 *     a queued, not-started request r on hotspot i with alternative j has
 *     benefit B = TTFT_{r,i} - TTFT_{r,j}, TTFT_{r,i} = work queued up to and
 *     including r, TTFT_{r,j} = W_j + c*(L - h_{r,j}); candidates sorted by
 *     (B desc, seq asc); migrate if B > 0 (re-evaluated with current W_j)
 *     and TTFT_{r,j} < SLO and j is live; stop once i is no longer a
 *     hotspot.  Single round; a request moves at most once per call.
 *
 *   Rebalancing variants (rebalance_flags): see OR_RB_* below.
 *
 *   Scaling (Sec. 3.4; App. A.1.3): add inserts V nodes per ring; remove
 *     deletes them, the instance keeps draining and takes no new work.
 *
 *   Adaptive hash-prefix length (Sec. 3.2, adapt_step_blocks > 0): see
 *     adapt_walk and adapt_window_end below (nodes named by the key of a
 *     prefix's last block; expand above 2T/n, drop below T/n per window).
 *
 *   Power of d choices (App. A.8): or_potc_max_loads below; routing with d
 *     candidates instead of two: or_route_batch_d below.
 *
 * Data structures are the obvious ones: sorted arrays rebuilt from scratch
 * on every membership change, an LRU as hash map + recency list, queues as
 * plain arrays.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

enum {
    OR_OK = 0, OR_ERR_INVALID_ARG = 1, OR_ERR_CAPACITY = 2, OR_ERR_NO_INSTANCES = 3,
    OR_ERR_DUPLICATE_ID = 4, OR_ERR_UNKNOWN_ID = 5, OR_ERR_ORDER = 6, OR_ERR_OOM = 9
};

/* ------------------------------------------------------------------ */
/* Published primitives                                                */
/* ------------------------------------------------------------------ */

/* SplitMix64 (Steele, Lea, Flood 2014): advance the state, return output. */
uint64_t or_splitmix64_next(uint64_t *state)
{
    uint64_t z = (*state += 0x9E3779B97F4A7C15ULL);
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
    return z ^ (z >> 31);
}

/* One SplitMix64 output step taken from state x (stateless mixer). */
uint64_t or_mix64(uint64_t x)
{
    uint64_t s = x;
    return or_splitmix64_next(&s);
}

/* MurmurHash3 64-bit finaliser (Appleby, public domain). */
uint64_t or_fmix64(uint64_t k)
{
    k ^= k >> 33;
    k *= 0xff51afd7ed558ccdULL;
    k ^= k >> 33;
    k *= 0xc4ceb9fe1a85ec53ULL;
    k ^= k >> 33;
    return k;
}

/* NH over one block of B tokens (B even) under key K. */
uint64_t or_nh(const uint32_t *t, const uint32_t *K, uint32_t B)
{
    uint64_t s = 0;
    for (uint32_t i = 0; i < B / 2; i++) {
        uint32_t a = t[2 * i] + K[2 * i];          /* mod 2^32 */
        uint32_t b = t[2 * i + 1] + K[2 * i + 1];  /* mod 2^32 */
        s += (uint64_t)a * (uint64_t)b;            /* mod 2^64 */
    }
    return s;
}

/* ------------------------------------------------------------------ */
/* Configuration and state                                             */
/* ------------------------------------------------------------------ */

typedef struct {
    uint32_t block_tokens;
    uint32_t route_prefix_blocks;
    uint32_t vnodes_per_instance;
    uint32_t max_instances;
    uint64_t cache_capacity_blocks;
    uint64_t slo_us;
    uint32_t cost_us_per_token;
    uint32_t hot_num, hot_den;
    uint32_t max_batch;
    uint64_t max_batch_tokens;
    uint64_t seed;
    uint32_t choice_rule;   /* OR_RULE_* */
    uint32_t adapt_step_blocks;   /* adaptive prefix: blocks per extension; 0 = fixed K_route */
    uint32_t adapt_max_blocks;    /* longest hash prefix, in blocks */
    uint32_t adapt_window;        /* non-empty batches per hotness window */
    uint32_t rebalance_flags;     /* OR_RB_* */
    uint32_t candidates;          /* rings (hash functions) kept: 0 or 2 = DualMap's two; up to OR_MAX_D */
} or_config;

#define OR_MAX_D 8

/* Rebalancing variants (the paper's own wording of Sec. 3.3 / App. A.1.2):
 * OR_RB_SLO_TARGET: an instance is overloaded when its queued work exceeds
 *   the SLO, and migration from it stops once its queued work is within the
 *   SLO ("until all requests in the overloaded instance's queue are
 *   expected to meet the TTFT SLO");
 * OR_RB_DOUBLE_OVERLOAD: a call migrates only after a routed batch in which
 *   some request's estimated TTFT exceeded the SLO on both candidates (the
 *   trigger "both candidate instances ... identified as overloaded");
 * OR_RB_FRESH_HITS: a migration candidate's TTFT on its other candidate j
 *   uses the hit found by probing j's cache as it stands at the rebalance
 *   call with the request's own block keys (the benefit's TTFT estimate
 *   queries the instance's KV metadata afresh), instead of the hit stored
 *   when the request was routed; queue entries keep their keys for this. */
enum { OR_RB_SLO_TARGET = 1, OR_RB_DOUBLE_OVERLOAD = 2, OR_RB_FRESH_HITS = 4 };

enum { OR_RULE_DUALMAP = 0, OR_RULE_CACHE_AFFINITY = 1, OR_RULE_LEAST_LOADED = 2,
       OR_RULE_MIN_TTFT = 3, OR_RULE_PREBLE = 4, OR_RULE_GLOBAL_CACHE_AFFINITY = 5,
       OR_RULE_GLOBAL_LEAST_LOADED = 6, OR_RULE_GLOBAL_MIN_TTFT = 7, OR_RULE_GLOBAL_PREBLE = 8 };

/* TTFT histogram: values 0..15 exact, then 16 buckets per power of two up
 * to 2^64. */
#define OR_HIST_BUCKETS 976

typedef struct {
    uint64_t key, stamp;
    int64_t newer, older;   /* recency list */
    int64_t chain;          /* bucket chain */
} lru_node;

typedef struct {
    lru_node *nodes;
    int64_t n_nodes, cap_nodes, free_head;
    int64_t *bucket;
    uint64_t nbucket;       /* power of two */
    int64_t mru, lru;
    uint64_t size;
} lru_t;

typedef struct {
    uint64_t seq;
    uint32_t L, c1, c2, h1, h2;
    uint64_t work, remaining;
    uint64_t moved_in_call;  /* rebalance call id that moved it here; 0 = none */
    uint64_t arrival;        /* batch time the request arrived with */
    uint64_t *keys;          /* OR_RB_FRESH_HITS: the prompt's block keys (owned), else NULL */
    uint32_t nblk;
} q_entry;

typedef struct {
    q_entry *e;
    uint64_t head, len, cap;  /* entries e[head .. head+len) */
} queue_t;

typedef struct {
    uint64_t pos;
    uint32_t id, v;
} vnode;

enum { INST_ABSENT = 0, INST_LIVE = 1, INST_DRAINING = 2 };

typedef struct {
    or_config cfg;
    uint32_t K1[64], K2[64];
    uint64_t G1, G2, Sc, Sr1, Sr2, Sv1, Sv2;
    /* functions f = 3..d of the d-candidate path: NH keys, salt, ring-position
     * and vnode seeds (index f - 3) */
    uint32_t Kx[OR_MAX_D - 2][64];
    uint64_t Gx[OR_MAX_D - 2], Srx[OR_MAX_D - 2], Svx[OR_MAX_D - 2];
    uint32_t nrings;    /* rings kept: max(2, candidates) */
    uint8_t *state;     /* per id: absent / live / draining */
    uint64_t *W;        /* queued work per id */
    queue_t *q;
    lru_t *cache;
    vnode *ring[OR_MAX_D];
    uint32_t ring_len;
    uint64_t clock, next_seq, t_prev;
    int have_time;
    uint64_t rebalance_calls;
    int both_over;      /* the last routed batch had a request over the SLO on both candidates */
    /* the last routed batch, kept for commit */
    uint32_t pend_n;
    uint64_t pend_seq0;
    uint32_t *pend_final, *pend_nblk;
    uint64_t **pend_keys;
    int pending;
    /* adaptive prefix: expanded nodes (sorted keys), this window's path
     * records (node key, depth), its requests and non-empty batches, and
     * the hash prefix length of each request of the last batch */
    uint64_t *ad_set;
    uint64_t ad_set_n;
    uint64_t *ad_rec_key;
    uint32_t *ad_rec_depth;
    uint64_t ad_rec_n, ad_rec_cap;
    uint64_t ad_requests, ad_batches;
    uint32_t *last_K;
    uint32_t last_n;
    /* metrics since create / the last reset */
    uint64_t m_requests, m_prompt_tokens, m_hit_tokens, m_switched, m_est_slo_met;
    uint64_t m_completed, m_ttft_sum, m_ttft_max, m_slo_met, m_batches;
    double m_cv_sum, m_cv_last;
    uint64_t m_hist[OR_HIST_BUCKETS];
} or_state;

/* ------------------------------------------------------------------ */
/* LRU: hash map key -> node, doubly linked recency list               */
/* ------------------------------------------------------------------ */

static uint64_t lru_bucket_of(const lru_t *c, uint64_t key)
{
    return (key ^ (key >> 29)) & (c->nbucket - 1);
}

static void lru_free(lru_t *c)
{
    free(c->nodes);
    free(c->bucket);
    memset(c, 0, sizeof *c);
}

static int lru_init(lru_t *c)
{
    memset(c, 0, sizeof *c);
    c->nbucket = 1024;
    c->bucket = (int64_t *)malloc(c->nbucket * sizeof(int64_t));
    if (!c->bucket) return OR_ERR_OOM;
    for (uint64_t i = 0; i < c->nbucket; i++) c->bucket[i] = -1;
    c->mru = c->lru = -1;
    c->free_head = -1;
    return OR_OK;
}

static int64_t lru_find(const lru_t *c, uint64_t key)
{
    int64_t i = c->bucket[lru_bucket_of(c, key)];
    while (i >= 0 && c->nodes[i].key != key) i = c->nodes[i].chain;
    return i;
}

static void lru_unlink(lru_t *c, int64_t i)
{
    lru_node *n = &c->nodes[i];
    if (n->newer >= 0) c->nodes[n->newer].older = n->older; else c->mru = n->older;
    if (n->older >= 0) c->nodes[n->older].newer = n->newer; else c->lru = n->newer;
    n->newer = n->older = -1;
}

static void lru_push_mru(lru_t *c, int64_t i)
{
    lru_node *n = &c->nodes[i];
    n->newer = -1;
    n->older = c->mru;
    if (c->mru >= 0) c->nodes[c->mru].newer = i;
    c->mru = i;
    if (c->lru < 0) c->lru = i;
}

static int lru_grow_buckets(lru_t *c)
{
    uint64_t nb = c->nbucket * 2;
    int64_t *b = (int64_t *)malloc(nb * sizeof(int64_t));
    if (!b) return OR_ERR_OOM;
    for (uint64_t i = 0; i < nb; i++) b[i] = -1;
    free(c->bucket);
    c->bucket = b;
    c->nbucket = nb;
    /* re-chain every live node (walk the recency list) */
    for (int64_t i = c->mru; i >= 0; i = c->nodes[i].older) {
        uint64_t h = lru_bucket_of(c, c->nodes[i].key);
        c->nodes[i].chain = c->bucket[h];
        c->bucket[h] = i;
    }
    return OR_OK;
}

static void lru_remove(lru_t *c, int64_t i)
{
    uint64_t h = lru_bucket_of(c, c->nodes[i].key);
    int64_t *link = &c->bucket[h];
    while (*link != i) link = &c->nodes[*link].chain;
    *link = c->nodes[i].chain;
    lru_unlink(c, i);
    c->nodes[i].chain = c->free_head;
    c->free_head = i;
    c->size--;
}

/* Touch `key` with `stamp` (insert if absent), then evict least recent
 * entries until at most `cap` remain.  This is the textbook LRU. */
static int lru_touch(lru_t *c, uint64_t key, uint64_t stamp, uint64_t cap)
{
    int64_t i = lru_find(c, key);
    if (i >= 0) {
        lru_unlink(c, i);
    } else {
        if (c->free_head >= 0) {
            i = c->free_head;
            c->free_head = c->nodes[i].chain;
        } else {
            if (c->n_nodes == c->cap_nodes) {
                int64_t nc = c->cap_nodes ? 2 * c->cap_nodes : 1024;
                lru_node *nn = (lru_node *)realloc(c->nodes, (size_t)nc * sizeof(lru_node));
                if (!nn) return OR_ERR_OOM;
                c->nodes = nn;
                c->cap_nodes = nc;
            }
            i = c->n_nodes++;
        }
        c->nodes[i].key = key;
        uint64_t h = lru_bucket_of(c, key);
        c->nodes[i].chain = c->bucket[h];
        c->bucket[h] = i;
        c->size++;
    }
    c->nodes[i].stamp = stamp;
    lru_push_mru(c, i);
    if (c->size > c->nbucket) {     /* rehash walks the recency list: after linking */
        int rc = lru_grow_buckets(c);
        if (rc) return rc;
    }
    while (c->size > cap) lru_remove(c, c->lru);
    return OR_OK;
}

static void lru_clear(lru_t *c)
{
    lru_free(c);
    lru_init(c);
}

/* ------------------------------------------------------------------ */
/* Key material, prompt hashing                                        */
/* ------------------------------------------------------------------ */

void or_derive_keys(uint64_t seed, uint32_t B, uint32_t *K1, uint32_t *K2, uint64_t *scalars)
{
    uint64_t s = seed;
    for (uint32_t j = 0; j < B; j++) K1[j] = (uint32_t)or_splitmix64_next(&s);
    for (uint32_t j = 0; j < B; j++) K2[j] = (uint32_t)or_splitmix64_next(&s);
    scalars[0] = or_splitmix64_next(&s) | 1ULL; /* G1 */
    scalars[1] = or_splitmix64_next(&s) | 1ULL; /* G2 */
    for (int j = 2; j < 7; j++) scalars[j] = or_splitmix64_next(&s); /* Sc Sr1 Sr2 Sv1 Sv2 */
}

/* All block keys of one prompt (n_blk of them) and its two ring positions.
 * Returns n_blk.  The per-block digests are summed in block order. */
static uint32_t prompt_keys(const or_state *s, const uint32_t *tok, uint32_t L,
                            uint64_t *keys, uint64_t *pos)
{
    const uint32_t B = s->cfg.block_tokens;
    const uint32_t nblk = L / B;
    uint32_t K = s->cfg.route_prefix_blocks < nblk ? s->cfg.route_prefix_blocks : nblk;
    uint64_t P1 = 0, P2 = 0;
    for (uint32_t k = 0; k < nblk; k++) {
        const uint32_t *t = tok + (uint64_t)k * B;
        uint64_t d1 = or_fmix64(or_nh(t, s->K1, B) + (uint64_t)(k + 1) * s->G1);
        P1 += d1;
        uint64_t key = or_fmix64(P1 ^ s->Sc);
        keys[k] = key ? key : 1;
        if (k < K) {
            uint64_t d2 = or_fmix64(or_nh(t, s->K2, B) + (uint64_t)(k + 1) * s->G2);
            P2 += d2;
            if (k == K - 1) {
                pos[0] = or_fmix64(P1 ^ s->Sr1);
                pos[1] = or_fmix64(P2 ^ s->Sr2);
            }
        }
    }
    return nblk;
}

/* ------------------------------------------------------------------ */
/* Rings                                                               */
/* ------------------------------------------------------------------ */

static int vnode_cmp(const void *a, const void *b)
{
    const vnode *x = (const vnode *)a, *y = (const vnode *)b;
    if (x->pos != y->pos) return x->pos < y->pos ? -1 : 1;
    if (x->id != y->id) return x->id < y->id ? -1 : 1;
    if (x->v != y->v) return x->v < y->v ? -1 : 1;
    return 0;
}

uint64_t or_vnode_pos(uint64_t Sv, uint32_t id, uint32_t v)
{
    return or_fmix64(or_mix64(((uint64_t)id << 32) | v) ^ Sv);
}

/* Index of the first entry with vpos >= p in a sorted array, 0 if none. */
uint32_t or_ring_successor(const uint64_t *vpos, uint32_t R, uint64_t p)
{
    uint32_t lo = 0, hi = R;          /* answer in [lo, hi] */
    while (lo < hi) {
        uint32_t mid = lo + (hi - lo) / 2;
        if (vpos[mid] < p) lo = mid + 1; else hi = mid;
    }
    return lo == R ? 0 : lo;
}

static uint32_t ring_owner(const or_state *s, int f, uint64_t p)
{
    /* binary search over the vnode records (same rule as or_ring_successor) */
    const vnode *r = s->ring[f];
    uint32_t lo = 0, hi = s->ring_len;
    while (lo < hi) {
        uint32_t mid = lo + (hi - lo) / 2;
        if (r[mid].pos < p) lo = mid + 1; else hi = mid;
    }
    return r[lo == s->ring_len ? 0 : lo].id;
}

static int rebuild_rings(or_state *s)
{
    uint32_t n = 0;
    for (uint32_t id = 0; id < s->cfg.max_instances; id++)
        if (s->state[id] == INST_LIVE) n++;
    uint32_t R = n * s->cfg.vnodes_per_instance;
    for (uint32_t f = 0; f < s->nrings; f++) {
        free(s->ring[f]);
        s->ring[f] = (vnode *)malloc((size_t)(R ? R : 1) * sizeof(vnode));
        if (!s->ring[f]) return OR_ERR_OOM;
        uint64_t Sv = f == 0 ? s->Sv1 : f == 1 ? s->Sv2 : s->Svx[f - 2];
        uint32_t k = 0;
        for (uint32_t id = 0; id < s->cfg.max_instances; id++) {
            if (s->state[id] != INST_LIVE) continue;
            for (uint32_t v = 0; v < s->cfg.vnodes_per_instance; v++) {
                s->ring[f][k].pos = or_vnode_pos(Sv, id, v);
                s->ring[f][k].id = id;
                s->ring[f][k].v = v;
                k++;
            }
        }
        qsort(s->ring[f], R, sizeof(vnode), vnode_cmp);
    }
    s->ring_len = R;
    return OR_OK;
}

static uint32_t n_live(const or_state *s)
{
    uint32_t n = 0;
    for (uint32_t id = 0; id < s->cfg.max_instances; id++) n += s->state[id] == INST_LIVE;
    return n;
}

/* Next live id after `id` in ascending order, cyclically. */
static uint32_t next_live_after(const or_state *s, uint32_t id)
{
    uint32_t M = s->cfg.max_instances;
    for (uint32_t k = 1; k <= M; k++) {
        uint32_t j = (id + k) % M;
        if (s->state[j] == INST_LIVE) return j;
    }
    return id;
}

/* ------------------------------------------------------------------ */
/* Queues                                                              */
/* ------------------------------------------------------------------ */

static int q_push(queue_t *q, const q_entry *x)
{
    if (q->head + q->len == q->cap) {
        if (q->head > 0) {  /* slide to the front */
            memmove(q->e, q->e + q->head, q->len * sizeof(q_entry));
            q->head = 0;
        }
        if (q->len == q->cap) {
            uint64_t nc = q->cap ? 2 * q->cap : 64;
            q_entry *ne = (q_entry *)realloc(q->e, nc * sizeof(q_entry));
            if (!ne) return OR_ERR_OOM;
            q->e = ne;
            q->cap = nc;
        }
    }
    q->e[q->head + q->len] = *x;
    q->len++;
    return OR_OK;
}

/* Remove the entry at position k (0 = head) keeping order. */
static void q_erase(queue_t *q, uint64_t k)
{
    q_entry *b = q->e + q->head;
    memmove(b + k, b + k + 1, (q->len - k - 1) * sizeof(q_entry));
    q->len--;
}

/* Run `delta` microseconds of prefill work off the head of the queue. */
/* Histogram bucket of a TTFT value: v < 16 is its own bucket; otherwise,
 * with e = floor(log2 v), bucket 16 + 16(e-4) + (the 4 bits below v's top
 * bit). */
uint32_t or_hist_bucket(uint64_t v)
{
    if (v < 16) return (uint32_t)v;
    uint32_t e = 63;
    while (!((v >> e) & 1)) e--;
    return 16 + 16 * (e - 4) + (uint32_t)((v >> (e - 4)) & 15);
}

/* Smallest value of bucket k. */
uint64_t or_hist_lower(uint32_t k)
{
    if (k < 16) return k;
    uint32_t e = 4 + (k - 16) / 16, sub = (k - 16) % 16;
    return (uint64_t)(16 + sub) << (e - 4);
}

static void record_ttft(or_state *s, uint64_t ttft)
{
    s->m_completed++;
    s->m_ttft_sum += ttft;
    if (ttft > s->m_ttft_max) s->m_ttft_max = ttft;
    if (ttft <= s->cfg.slo_us) s->m_slo_met++;
    s->m_hist[or_hist_bucket(ttft)]++;
}

/* Run `delta` us of instance id's queue, the window starting at t0. */
static void q_drain(or_state *s, uint32_t id, uint64_t delta, uint64_t t0)
{
    queue_t *q = &s->q[id];
    uint64_t run = 0;   /* work finished since t0 */
    while (q->len > 0) {
        q_entry *h = &q->e[q->head];
        if (h->remaining <= delta - run) {
            run += h->remaining;
            s->W[id] -= h->remaining;
            record_ttft(s, t0 + run - h->arrival);
            free(h->keys);
            q->head++;
            q->len--;
        } else {
            h->remaining -= delta - run;
            s->W[id] -= delta - run;
            break;
        }
    }
    if (q->len == 0) q->head = 0;
}

/* ------------------------------------------------------------------ */
/* Lifecycle                                                           */
/* ------------------------------------------------------------------ */

static void clear_pending(or_state *s)
{
    if (s->pend_keys)
        for (uint32_t i = 0; i < s->pend_n; i++) free(s->pend_keys[i]);
    free(s->pend_keys);
    free(s->pend_final);
    free(s->pend_nblk);
    s->pend_keys = NULL;
    s->pend_final = s->pend_nblk = NULL;
    s->pend_n = 0;
    s->pending = 0;
}

void or_destroy(or_state *s)
{
    if (!s) return;
    clear_pending(s);
    for (uint32_t i = 0; i < s->cfg.max_instances; i++) {
        if (s->cache) lru_free(&s->cache[i]);
        if (s->q) {
            for (uint64_t k = 0; k < s->q[i].len; k++) free(s->q[i].e[s->q[i].head + k].keys);
            free(s->q[i].e);
        }
    }
    free(s->cache);
    free(s->q);
    free(s->W);
    free(s->state);
    for (uint32_t f = 0; f < OR_MAX_D; f++) free(s->ring[f]);
    free(s->ad_set);
    free(s->ad_rec_key);
    free(s->ad_rec_depth);
    free(s->last_K);
    free(s);
}

int or_create(const or_config *cfg, or_state **out)
{
    *out = NULL;
    uint32_t B = cfg->block_tokens;
    if (B < 2 || B > 64 || (B & 1) || cfg->route_prefix_blocks < 1 || cfg->choice_rule > OR_RULE_GLOBAL_PREBLE ||
        cfg->vnodes_per_instance < 1 || cfg->max_instances < 2 ||
        cfg->cache_capacity_blocks < 1 || cfg->cost_us_per_token < 1 ||
        cfg->hot_den < 1 || cfg->max_batch < 1 || cfg->max_batch_tokens < B)
        return OR_ERR_INVALID_ARG;
    if (cfg->adapt_step_blocks &&
        (cfg->adapt_max_blocks <= cfg->route_prefix_blocks || cfg->adapt_max_blocks > 2048 ||
         cfg->adapt_window < 1))
        return OR_ERR_INVALID_ARG;
    if (cfg->candidates > OR_MAX_D) return OR_ERR_INVALID_ARG;
    or_state *s = (or_state *)calloc(1, sizeof(or_state));
    if (!s) return OR_ERR_OOM;
    s->cfg = *cfg;
    uint64_t sc[7];
    or_derive_keys(cfg->seed, B, s->K1, s->K2, sc);
    s->G1 = sc[0]; s->G2 = sc[1]; s->Sc = sc[2]; s->Sr1 = sc[3]; s->Sr2 = sc[4];
    s->Sv1 = sc[5]; s->Sv2 = sc[6];
    /* functions 3..d continue the same SplitMix64 stream after DualMap's
     * nine draws, so two functions keep exactly DualMap's key material */
    {
        uint64_t st = cfg->seed;
        for (uint32_t j = 0; j < 2 * B + 7; j++) or_splitmix64_next(&st);
        for (uint32_t f = 0; f + 2 < OR_MAX_D; f++) {
            for (uint32_t j = 0; j < B; j++) s->Kx[f][j] = (uint32_t)or_splitmix64_next(&st);
            s->Gx[f] = or_splitmix64_next(&st) | 1ULL;
            s->Srx[f] = or_splitmix64_next(&st);
            s->Svx[f] = or_splitmix64_next(&st);
        }
    }
    s->nrings = cfg->candidates > 2 ? cfg->candidates : 2;
    uint32_t M = cfg->max_instances;
    s->state = (uint8_t *)calloc(M, 1);
    s->W = (uint64_t *)calloc(M, sizeof(uint64_t));
    s->q = (queue_t *)calloc(M, sizeof(queue_t));
    s->cache = (lru_t *)calloc(M, sizeof(lru_t));
    if (!s->state || !s->W || !s->q || !s->cache) { or_destroy(s); return OR_ERR_OOM; }
    for (uint32_t i = 0; i < M; i++)
        if (lru_init(&s->cache[i])) { or_destroy(s); return OR_ERR_OOM; }
    if (rebuild_rings(s)) { or_destroy(s); return OR_ERR_OOM; }
    *out = s;
    return OR_OK;
}

int or_add_instance(or_state *s, uint32_t id)
{
    if (id >= s->cfg.max_instances) return OR_ERR_INVALID_ARG;
    if (s->state[id] == INST_LIVE) return OR_ERR_DUPLICATE_ID;
    if (s->state[id] == INST_DRAINING && s->q[id].len > 0) return OR_ERR_DUPLICATE_ID;
    s->state[id] = INST_LIVE;
    lru_clear(&s->cache[id]);   /* a (re-)added instance starts with an empty index */
    s->W[id] = 0;
    return rebuild_rings(s);
}

int or_remove_instance(or_state *s, uint32_t id)
{
    if (id >= s->cfg.max_instances || s->state[id] != INST_LIVE) return OR_ERR_UNKNOWN_ID;
    s->state[id] = INST_DRAINING;
    return rebuild_rings(s);
}

/* ------------------------------------------------------------------ */
/* The routing step                                                     */
/* ------------------------------------------------------------------ */

/* Cache affinity: more hits; equal hits, the less-loaded (tie c1). */
static uint32_t choose_affinity(uint32_t c1, uint32_t c2, uint32_t h1, uint32_t h2,
                                uint64_t W1, uint64_t W2)
{
    if (h1 != h2) return h1 > h2 ? c1 : c2;
    return W2 < W1 ? c2 : c1;
}

/* The choice between the two candidates under `rule` (Sec. 3.2 for
 * DualMap's SLO-aware rule; the compared rules as listed in the header).
 * Returns the chosen id; *switched is set when the SLO rule overrode cache
 * affinity (DualMap) or when the candidate with fewer hits was chosen
 * (other rules). */
uint32_t or_choose(uint32_t rule, uint32_t c1, uint32_t c2, uint32_t h1, uint32_t h2, uint32_t L,
                   uint64_t W1, uint64_t W2, uint64_t slo, uint32_t cost,
                   uint64_t *ttft1, uint64_t *ttft2, uint8_t *switched)
{
    *ttft1 = W1 + (uint64_t)cost * (L - h1);
    *ttft2 = W2 + (uint64_t)cost * (L - h2);
    *switched = 0;
    if (rule != OR_RULE_DUALMAP) {
        uint32_t ch;
        uint32_t hmax = h1 > h2 ? h1 : h2;
        if (rule == OR_RULE_GLOBAL_CACHE_AFFINITY) return c1;
        if (rule == OR_RULE_CACHE_AFFINITY ||
            (rule == OR_RULE_PREBLE && 2 * (uint64_t)hmax > L))
            ch = choose_affinity(c1, c2, h1, h2, W1, W2);
        else if (rule == OR_RULE_LEAST_LOADED)
            ch = W2 < W1 ? c2 : c1;
        else   /* min TTFT, and Preble below half the prompt */
            ch = *ttft2 < *ttft1 ? c2 : c1;
        uint32_t h_ch = ch == c1 ? h1 : h2, h_other = ch == c1 ? h2 : h1;
        *switched = h_ch < h_other;
        return ch;
    }
    if (h1 == h2) return W2 < W1 ? c2 : c1;
    int a_is_1 = h1 > h2;
    uint64_t ttft_a = a_is_1 ? *ttft1 : *ttft2;
    uint64_t Wa = a_is_1 ? W1 : W2, Wb = a_is_1 ? W2 : W1;
    uint32_t a = a_is_1 ? c1 : c2, b = a_is_1 ? c2 : c1;
    if (ttft_a <= slo) return a;
    *switched = 1;
    return Wb < Wa ? b : a;
}

static double u128_to_double(unsigned __int128 x)
{
    return (double)(uint64_t)(x >> 64) * 18446744073709551616.0 + (double)(uint64_t)x;
}

/* Coefficient of variation of the live instances' queued work (Sec. 2.2). */
static double load_cv(const or_state *s)
{
    unsigned __int128 S1 = 0, S2 = 0;
    uint64_t n = 0;
    for (uint32_t id = 0; id < s->cfg.max_instances; id++)
        if (s->state[id] == INST_LIVE) {
            S1 += s->W[id];
            S2 += (unsigned __int128)s->W[id] * s->W[id];
            n++;
        }
    if (S1 == 0) return 0.0;
    return sqrt(u128_to_double(n * S2 - S1 * S1)) / u128_to_double(S1);
}

/* The rules over all live instances (see the header); h[id] = hit tokens
 * of the request on instance id. */
static uint32_t choose_global(const or_state *s, uint32_t rule, const uint32_t *h, uint32_t L)
{
    const uint64_t cost = s->cfg.cost_us_per_token;
    uint32_t hmax = 0;
    for (uint32_t id = 0; id < s->cfg.max_instances; id++)
        if (s->state[id] == INST_LIVE && h[id] > hmax) hmax = h[id];
    const int affine = rule == OR_RULE_GLOBAL_PREBLE && 2 * (uint64_t)hmax > L;
    uint32_t best = UINT32_MAX;
    uint64_t best_key = 0;
    for (uint32_t id = 0; id < s->cfg.max_instances; id++) {
        if (s->state[id] != INST_LIVE) continue;
        uint64_t key;
        if (rule == OR_RULE_GLOBAL_LEAST_LOADED) {
            key = s->W[id];
        } else if (affine) {
            if (h[id] != hmax) continue;
            key = s->W[id];
        } else {
            key = s->W[id] + cost * (L - h[id]);
        }
        if (best == UINT32_MAX || key < best_key) { best = id; best_key = key; }
    }
    return best;
}

/* ------------------------------------------------------------------ */
/* Adaptive hash-prefix length (Sec. 3.2, "how long prefix")            */
/* ------------------------------------------------------------------ */

/* Ring positions of a prompt hashed over its first K blocks. */
static void positions_for(const or_state *s, const uint32_t *tok, uint32_t K, uint64_t *pos)
{
    const uint32_t B = s->cfg.block_tokens;
    uint64_t P1 = 0, P2 = 0;
    for (uint32_t k = 0; k < K; k++) {
        const uint32_t *t = tok + (uint64_t)k * B;
        P1 += or_fmix64(or_nh(t, s->K1, B) + (uint64_t)(k + 1) * s->G1);
        P2 += or_fmix64(or_nh(t, s->K2, B) + (uint64_t)(k + 1) * s->G2);
    }
    pos[0] = or_fmix64(P1 ^ s->Sr1);
    pos[1] = or_fmix64(P2 ^ s->Sr2);
}

static int cmp_u64(const void *a, const void *b)
{
    uint64_t x = *(const uint64_t *)a, y = *(const uint64_t *)b;
    return x < y ? -1 : x > y;
}

static int expanded(const or_state *s, uint64_t key)
{
    return s->ad_set_n && bsearch(&key, s->ad_set, s->ad_set_n, sizeof(uint64_t), cmp_u64) != NULL;
}

static int path_push(or_state *s, uint64_t key, uint32_t depth)
{
    if (s->ad_rec_n == s->ad_rec_cap) {
        uint64_t nc = s->ad_rec_cap ? 2 * s->ad_rec_cap : 1024;
        uint64_t *k = (uint64_t *)realloc(s->ad_rec_key, nc * sizeof(uint64_t));
        if (!k) return OR_ERR_OOM;
        s->ad_rec_key = k;
        uint32_t *d = (uint32_t *)realloc(s->ad_rec_depth, nc * sizeof(uint32_t));
        if (!d) return OR_ERR_OOM;
        s->ad_rec_depth = d;
        s->ad_rec_cap = nc;
    }
    s->ad_rec_key[s->ad_rec_n] = key;
    s->ad_rec_depth[s->ad_rec_n] = depth;
    s->ad_rec_n++;
    return OR_OK;
}

/* The request's hash prefix length: start at min(K_route, n_blk) blocks;
 * while the node of the current prefix (the key of its last block) is
 * expanded and the prompt and the cap allow, extend by one step.  Every
 * node on the way is recorded for this window's hotness counts. */
static int adapt_walk(or_state *s, const uint64_t *keys, uint32_t nblk, uint32_t *K)
{
    const or_config *c = &s->cfg;
    uint32_t d = c->route_prefix_blocks < nblk ? c->route_prefix_blocks : nblk;
    int rc = path_push(s, keys[d - 1], d);
    while (!rc && d < nblk && d < c->adapt_max_blocks && expanded(s, keys[d - 1])) {
        d += c->adapt_step_blocks;
        if (d > nblk) d = nblk;
        if (d > c->adapt_max_blocks) d = c->adapt_max_blocks;
        rc = path_push(s, keys[d - 1], d);
    }
    *K = d;
    return rc;
}

static int cmp_rec(const void *a, const void *b)
{
    const uint64_t *x = (const uint64_t *)a, *y = (const uint64_t *)b;
    return x[0] < y[0] ? -1 : x[0] > y[0];
}

/* End of a window: with n live instances and T requests in the window, a
 * node not expanded becomes expanded when its share count/T > 2/n and it
 * lies above the cap; an expanded node stays expanded unless count/T < 1/n
 * (so nodes no request reached are dropped).  Counts then restart. */
static int adapt_window_end(or_state *s)
{
    const uint64_t n = n_live(s), T = s->ad_requests;
    uint64_t m = s->ad_rec_n;
    uint64_t *rec = (uint64_t *)malloc((m ? m : 1) * 2 * sizeof(uint64_t));
    uint64_t *next = (uint64_t *)malloc((s->ad_set_n + m + 1) * sizeof(uint64_t));
    if (!rec || !next) { free(rec); free(next); return OR_ERR_OOM; }
    for (uint64_t i = 0; i < m; i++) {
        rec[2 * i] = s->ad_rec_key[i];
        rec[2 * i + 1] = s->ad_rec_depth[i];
    }
    qsort(rec, m, 2 * sizeof(uint64_t), cmp_rec);
    uint64_t nn = 0;
    /* expanded nodes: kept unless cold */
    for (uint64_t j = 0; j < s->ad_set_n; j++) {
        uint64_t key = s->ad_set[j], count = 0;
        for (uint64_t i = 0; i < m; i++)
            if (rec[2 * i] == key) count++;
        if (!(count * n < T)) next[nn++] = key;
    }
    /* nodes reached this window: expanded when hot */
    for (uint64_t i = 0; i < m;) {
        uint64_t e = i;
        while (e < m && rec[2 * e] == rec[2 * i]) e++;
        const uint64_t key = rec[2 * i], depth = rec[2 * i + 1], count = e - i;
        if (!expanded(s, key) && depth < s->cfg.adapt_max_blocks && count * n > 2 * T) next[nn++] = key;
        i = e;
    }
    qsort(next, nn, sizeof(uint64_t), cmp_u64);
    free(rec);
    free(s->ad_set);
    s->ad_set = next;
    s->ad_set_n = nn;
    s->ad_rec_n = 0;
    s->ad_requests = 0;
    s->ad_batches = 0;
    return OR_OK;
}

static uint32_t leading_hits(const lru_t *c, const uint64_t *keys, uint32_t nblk)
{
    uint32_t m = 0;
    while (m < nblk && lru_find(c, keys[m]) >= 0) m++;
    return m;
}

/* The start of a routed batch: argument checks, the queues drain for the
 * elapsed time (Sec. 3.2 load = pending prefill), and the pending-commit
 * arrays for n requests (keys filled in by the caller). */
static int route_prologue(or_state *s, const uint32_t *lengths, uint32_t n, uint64_t t_batch)
{
    const or_config *cf = &s->cfg;
    if (n > cf->max_batch) return OR_ERR_CAPACITY;
    if (n_live(s) < 2) return OR_ERR_NO_INSTANCES;
    if (s->have_time && t_batch < s->t_prev) return OR_ERR_ORDER;
    uint64_t total = 0;
    for (uint32_t r = 0; r < n; r++) {
        if (lengths[r] < cf->block_tokens) return OR_ERR_INVALID_ARG;
        total += lengths[r];
    }
    if (total > cf->max_batch_tokens) return OR_ERR_CAPACITY;

    /* time advances; every instance's queue runs for the elapsed us */
    uint64_t delta = s->have_time ? t_batch - s->t_prev : 0;
    for (uint32_t id = 0; id < cf->max_instances; id++)
        if (s->state[id] != INST_ABSENT) q_drain(s, id, delta, s->t_prev);
    s->t_prev = t_batch;
    s->have_time = 1;

    clear_pending(s);
    s->pend_n = n;
    s->pend_seq0 = s->next_seq;
    s->pend_final = (uint32_t *)malloc((n ? n : 1) * sizeof(uint32_t));
    s->pend_nblk = (uint32_t *)malloc((n ? n : 1) * sizeof(uint32_t));
    s->pend_keys = (uint64_t **)calloc(n ? n : 1, sizeof(uint64_t *));
    uint32_t *lk = (uint32_t *)realloc(s->last_K, (n ? n : 1) * sizeof(uint32_t));
    if (!lk) return OR_ERR_OOM;
    s->last_K = lk;
    s->last_n = n;
    if (!s->pend_final || !s->pend_nblk || !s->pend_keys) return OR_ERR_OOM;
    return OR_OK;
}

static int route_choose(or_state *s, const uint32_t *lengths, uint32_t n, uint64_t t_batch,
                        const uint32_t *cand1, const uint32_t *cand2, const uint32_t *hit1, const uint32_t *hit2,
                        const uint32_t *hall, uint64_t *ttft1, uint64_t *ttft2, uint32_t *chosen,
                        uint8_t *switched);

int or_route_batch(or_state *s, const uint32_t *tokens, const uint64_t *offsets,
                   const uint32_t *lengths, uint32_t n, uint64_t t_batch,
                   uint32_t *cand1, uint32_t *cand2, uint32_t *hit1, uint32_t *hit2,
                   uint64_t *ttft1, uint64_t *ttft2, uint32_t *chosen, uint8_t *switched)
{
    const or_config *cf = &s->cfg;
    int rc0 = route_prologue(s, lengths, n, t_batch);
    if (rc0) return rc0;

    /* hits on every live instance, for the rules that look at all of them */
    uint32_t *hall = NULL;
    if (cf->choice_rule >= OR_RULE_GLOBAL_LEAST_LOADED) {
        hall = (uint32_t *)malloc(((size_t)n * cf->max_instances + 1) * sizeof(uint32_t));
        if (!hall) return OR_ERR_OOM;
    }

    /* 1) hash, ring lookup, distinct fix, probes: all against batch-start state */
    for (uint32_t r = 0; r < n; r++) {
        uint32_t L = lengths[r];
        uint64_t *keys = (uint64_t *)malloc((size_t)(L / cf->block_tokens) * sizeof(uint64_t));
        if (!keys) return OR_ERR_OOM;
        uint64_t pos[2];
        uint32_t nblk = prompt_keys(s, tokens + offsets[r], L, keys, pos);
        uint32_t K = cf->route_prefix_blocks < nblk ? cf->route_prefix_blocks : nblk;
        if (cf->adapt_step_blocks) {
            int rc = adapt_walk(s, keys, nblk, &K);
            if (rc) return rc;
            if (K != (cf->route_prefix_blocks < nblk ? cf->route_prefix_blocks : nblk))
                positions_for(s, tokens + offsets[r], K, pos);
        }
        s->last_K[r] = K;
        s->pend_keys[r] = keys;
        s->pend_nblk[r] = nblk;
        uint32_t c1 = ring_owner(s, 0, pos[0]);
        uint32_t c2 = ring_owner(s, 1, pos[1]);
        if (c2 == c1) c2 = next_live_after(s, c1);
        cand1[r] = c1;
        cand2[r] = c2;
        hit1[r] = cf->block_tokens * leading_hits(&s->cache[c1], keys, nblk);
        hit2[r] = cf->block_tokens * leading_hits(&s->cache[c2], keys, nblk);
        if (hall)
            for (uint32_t id = 0; id < cf->max_instances; id++)
                hall[(size_t)r * cf->max_instances + id] =
                    s->state[id] == INST_LIVE ? cf->block_tokens * leading_hits(&s->cache[id], keys, nblk) : 0;
    }
    int rc2 = route_choose(s, lengths, n, t_batch, cand1, cand2, hit1, hit2, hall, ttft1, ttft2, chosen, switched);
    free(hall);
    if (rc2) return rc2;
    if (cf->adapt_step_blocks && n > 0) {
        s->ad_requests += n;
        if (++s->ad_batches == cf->adapt_window) {
            int rc = adapt_window_end(s);
            if (rc) return rc;
        }
    }
    s->pending = 1;
    return OR_OK;
}

/* The choice half of a routed batch (Sec. 3.2 "SLO-Aware Strategy"): in
 * arrival order each request's TTFT estimates, its choice (hall: hits on
 * every instance, for the cluster-wide rules, else NULL), its queue entry
 * and the loads, the metrics; then the batch's CV sample. */
static int route_choose(or_state *s, const uint32_t *lengths, uint32_t n, uint64_t t_batch,
                        const uint32_t *cand1, const uint32_t *cand2, const uint32_t *hit1, const uint32_t *hit2,
                        const uint32_t *hall, uint64_t *ttft1, uint64_t *ttft2, uint32_t *chosen,
                        uint8_t *switched)
{
    const or_config *cf = &s->cfg;
    /* 2) choices in arrival order; loads update as we go */
    s->both_over = 0;
    for (uint32_t r = 0; r < n; r++) {
        uint32_t c1 = cand1[r], c2 = cand2[r];
        uint32_t ch, hch;
        if (hall) {
            const uint32_t *h = hall + (size_t)r * cf->max_instances;
            ch = choose_global(s, cf->choice_rule, h, lengths[r]);
            ttft1[r] = s->W[c1] + (uint64_t)cf->cost_us_per_token * (lengths[r] - hit1[r]);
            ttft2[r] = s->W[c2] + (uint64_t)cf->cost_us_per_token * (lengths[r] - hit2[r]);
            switched[r] = 0;
            hch = h[ch];
        } else {
            ch = or_choose(cf->choice_rule, c1, c2, hit1[r], hit2[r], lengths[r], s->W[c1], s->W[c2],
                           cf->slo_us, cf->cost_us_per_token, &ttft1[r], &ttft2[r], &switched[r]);
            hch = ch == c1 ? hit1[r] : hit2[r];
        }
        chosen[r] = ch;
        if (ttft1[r] > cf->slo_us && ttft2[r] > cf->slo_us) s->both_over = 1;
        q_entry e;
        e.seq = s->next_seq++;
        e.L = lengths[r]; e.c1 = c1; e.c2 = c2; e.h1 = hit1[r]; e.h2 = hit2[r];
        e.work = e.remaining = (uint64_t)cf->cost_us_per_token * (lengths[r] - hch);
        e.moved_in_call = 0;
        e.arrival = t_batch;
        e.keys = NULL;
        e.nblk = s->pend_nblk[r];
        if ((cf->rebalance_flags & OR_RB_FRESH_HITS) && e.nblk) {
            e.keys = (uint64_t *)malloc((size_t)e.nblk * sizeof(uint64_t));
            if (!e.keys) return OR_ERR_OOM;
            memcpy(e.keys, s->pend_keys[r], (size_t)e.nblk * sizeof(uint64_t));
        }
        if (q_push(&s->q[ch], &e)) { free(e.keys); return OR_ERR_OOM; }
        s->W[ch] += e.work;
        s->pend_final[r] = ch;
        s->m_requests++;
        s->m_prompt_tokens += lengths[r];
        s->m_hit_tokens += hch;
        s->m_switched += switched[r];
        s->m_est_slo_met += s->W[ch] <= cf->slo_us;   /* the load including this request */
    }
    if (n > 0) {
        s->m_cv_last = load_cv(s);
        s->m_cv_sum += s->m_cv_last;
        s->m_batches++;
    }
    return OR_OK;
}

/* Sharded routing, the per-rank half (the multi-GPU split of the routing
 * step; no paper counterpart): for requests r0 .. r1-1 of a batch, their
 * block keys, hash length, candidates and hits, against the state as it
 * stands (the batch's start: nothing here changes the state).  keys gets
 * every request's keys, request after request (at most key_cap).  The
 * fixed prefix length and the pair rules only. */
int or_route_part(or_state *s, const uint32_t *tokens, const uint64_t *offsets, const uint32_t *lengths,
                  uint32_t r0, uint32_t r1, uint32_t *K, uint32_t *cand1, uint32_t *cand2, uint32_t *hit1,
                  uint32_t *hit2, uint64_t *keys, uint64_t key_cap)
{
    const or_config *cf = &s->cfg;
    if (cf->adapt_step_blocks || cf->choice_rule >= OR_RULE_GLOBAL_LEAST_LOADED || r0 > r1) return OR_ERR_INVALID_ARG;
    if (n_live(s) < 2) return OR_ERR_NO_INSTANCES;
    uint64_t used = 0;
    for (uint32_t r = r0; r < r1; r++) {
        if (lengths[r] < cf->block_tokens) return OR_ERR_INVALID_ARG;
        const uint32_t nb = lengths[r] / cf->block_tokens;
        if (used + nb > key_cap) return OR_ERR_CAPACITY;
        uint64_t pos[2];
        uint32_t nblk = prompt_keys(s, tokens + offsets[r], lengths[r], keys + used, pos);
        const uint32_t k = r - r0;
        K[k] = cf->route_prefix_blocks < nblk ? cf->route_prefix_blocks : nblk;
        uint32_t c1 = ring_owner(s, 0, pos[0]);
        uint32_t c2 = ring_owner(s, 1, pos[1]);
        if (c2 == c1) c2 = next_live_after(s, c1);
        cand1[k] = c1;
        cand2[k] = c2;
        hit1[k] = cf->block_tokens * leading_hits(&s->cache[c1], keys + used, nblk);
        hit2[k] = cf->block_tokens * leading_hits(&s->cache[c2], keys + used, nblk);
        used += nblk;
    }
    return OR_OK;
}

/* Sharded routing, the replicated half: the batch routed with every
 * request's keys, hash length, candidates and hits given (gathered from
 * the ranks' or_route_part): the same drain, choices, queues, metrics and
 * pending commit as or_route_batch. */
int or_route_given(or_state *s, const uint32_t *lengths, uint32_t n, uint64_t t_batch, const uint32_t *K,
                   const uint32_t *cand1, const uint32_t *cand2, const uint32_t *hit1, const uint32_t *hit2,
                   const uint64_t *keys, uint64_t *ttft1, uint64_t *ttft2, uint32_t *chosen, uint8_t *switched)
{
    const or_config *cf = &s->cfg;
    if (cf->adapt_step_blocks || cf->choice_rule >= OR_RULE_GLOBAL_LEAST_LOADED) return OR_ERR_INVALID_ARG;
    int rc = route_prologue(s, lengths, n, t_batch);
    if (rc) return rc;
    uint64_t used = 0;
    for (uint32_t r = 0; r < n; r++) {
        const uint32_t nb = lengths[r] / cf->block_tokens;
        uint64_t *k = (uint64_t *)malloc((size_t)(nb ? nb : 1) * sizeof(uint64_t));
        if (!k) return OR_ERR_OOM;
        memcpy(k, keys + used, (size_t)nb * sizeof(uint64_t));
        used += nb;
        s->pend_keys[r] = k;
        s->pend_nblk[r] = nb;
        s->last_K[r] = K[r];
    }
    rc = route_choose(s, lengths, n, t_batch, cand1, cand2, hit1, hit2, NULL, ttft1, ttft2, chosen, switched);
    if (rc) return rc;
    s->pending = 1;
    return OR_OK;
}

/* ------------------------------------------------------------------ */
/* d candidates (App. A.8, "Optimal Candidate Set Size")                */
/* ------------------------------------------------------------------ */

/* The generalisation of the routing step that App. A.8 weighs: d
 * independent hash functions of the prompt prefix, d rings, d candidates,
 * d probes, one choice.  Function f's ring position is
 * fmix64(P^f_{K-1} xor S_rf) with P^f the chained sum of its block digests,
 * as for f = 1, 2; functions 3..d draw their key material after DualMap's.
 * Distinct candidates: c_1 = the owner on ring 1; c_f (f >= 2) = the owner on
 * ring f unless an earlier candidate has it, then the next live id after
 * that owner, in ascending order, cyclically, that is not yet a candidate
 * (for d = 2 this is DualMap's rule).  Choice, DualMap's rule over d
 * candidates (a reading: the paper states it for two): among the
 * candidates with the most hit tokens, a is the less loaded by W (tie: the
 * earlier f); a is chosen if every candidate has that many hits or
 * ttft_a <= SLO; otherwise the least loaded candidate by W (tie: a, then the
 * earlier f), and the request is flagged "switched" (as DualMap flags it,
 * even when that candidate is a itself).  d = 2 is DualMap's rule;
 * d = 1 always takes the ring-1 owner, i.e. cache affinity.  Loads, queues,
 * metrics and the commit are those of or_route_batch (queue entries keep
 * the first two candidates; rebalancing is defined for d = 2 only).
 * cand, hit, ttft hold n*d entries (request-major). */
static uint64_t ring_pos_f(const or_state *s, const uint32_t *tok, uint32_t K, uint32_t f)
{
    const uint32_t B = s->cfg.block_tokens;
    const uint32_t *Kf = f == 0 ? s->K1 : f == 1 ? s->K2 : s->Kx[f - 2];
    const uint64_t G = f == 0 ? s->G1 : f == 1 ? s->G2 : s->Gx[f - 2];
    const uint64_t Sr = f == 0 ? s->Sr1 : f == 1 ? s->Sr2 : s->Srx[f - 2];
    uint64_t P = 0;
    for (uint32_t k = 0; k < K; k++) P += or_fmix64(or_nh(tok + (uint64_t)k * B, Kf, B) + (uint64_t)(k + 1) * G);
    return or_fmix64(P ^ Sr);
}

int or_route_batch_d(or_state *s, uint32_t d, const uint32_t *tokens, const uint64_t *offsets,
                     const uint32_t *lengths, uint32_t n, uint64_t t_batch, uint32_t *cand, uint32_t *hit,
                     uint64_t *ttft, uint32_t *chosen, uint8_t *switched)
{
    const or_config *cf = &s->cfg;
    if (d < 1 || d > s->nrings || cf->adapt_step_blocks || cf->choice_rule != OR_RULE_DUALMAP)
        return OR_ERR_INVALID_ARG;
    if (n > cf->max_batch) return OR_ERR_CAPACITY;
    if (n_live(s) < 2 || n_live(s) < d) return OR_ERR_NO_INSTANCES;
    if (s->have_time && t_batch < s->t_prev) return OR_ERR_ORDER;
    uint64_t total = 0;
    for (uint32_t r = 0; r < n; r++) {
        if (lengths[r] < cf->block_tokens) return OR_ERR_INVALID_ARG;
        total += lengths[r];
    }
    if (total > cf->max_batch_tokens) return OR_ERR_CAPACITY;
    uint64_t delta = s->have_time ? t_batch - s->t_prev : 0;
    for (uint32_t id = 0; id < cf->max_instances; id++)
        if (s->state[id] != INST_ABSENT) q_drain(s, id, delta, s->t_prev);
    s->t_prev = t_batch;
    s->have_time = 1;
    clear_pending(s);
    s->pend_n = n;
    s->pend_seq0 = s->next_seq;
    s->pend_final = (uint32_t *)malloc((n ? n : 1) * sizeof(uint32_t));
    s->pend_nblk = (uint32_t *)malloc((n ? n : 1) * sizeof(uint32_t));
    s->pend_keys = (uint64_t **)calloc(n ? n : 1, sizeof(uint64_t *));
    uint32_t *lk = (uint32_t *)realloc(s->last_K, (n ? n : 1) * sizeof(uint32_t));
    if (!lk) return OR_ERR_OOM;
    s->last_K = lk;
    s->last_n = n;
    if (!s->pend_final || !s->pend_nblk || !s->pend_keys) return OR_ERR_OOM;
    /* 1) hash, d ring lookups, distinct fix, d probes (batch-start state) */
    for (uint32_t r = 0; r < n; r++) {
        const uint32_t L = lengths[r];
        const uint32_t *tok = tokens + offsets[r];
        uint64_t *keys = (uint64_t *)malloc((size_t)(L / cf->block_tokens) * sizeof(uint64_t));
        if (!keys) return OR_ERR_OOM;
        uint64_t pos2[2];
        const uint32_t nblk = prompt_keys(s, tok, L, keys, pos2);
        const uint32_t K = cf->route_prefix_blocks < nblk ? cf->route_prefix_blocks : nblk;
        s->last_K[r] = K;
        s->pend_keys[r] = keys;
        s->pend_nblk[r] = nblk;
        uint32_t *c = cand + (size_t)r * d;
        for (uint32_t f = 0; f < d; f++) {
            uint32_t x = ring_owner(s, (int)f, ring_pos_f(s, tok, K, f));
            for (;;) {   /* taken by an earlier candidate: the next live id after it */
                uint32_t taken = 0;
                for (uint32_t g = 0; g < f; g++) taken |= c[g] == x;
                if (!taken) break;
                x = next_live_after(s, x);
            }
            c[f] = x;
            hit[(size_t)r * d + f] = cf->block_tokens * leading_hits(&s->cache[x], keys, nblk);
        }
    }
    /* 2) choices in arrival order */
    s->both_over = 0;
    for (uint32_t r = 0; r < n; r++) {
        const uint32_t *c = cand + (size_t)r * d, *h = hit + (size_t)r * d;
        const uint32_t L = lengths[r];
        uint32_t hmax = 0, nmax = 0;
        for (uint32_t f = 0; f < d; f++) hmax = h[f] > hmax ? h[f] : hmax;
        uint32_t a = d;
        int all_over = 1;
        for (uint32_t f = 0; f < d; f++) {
            ttft[(size_t)r * d + f] = s->W[c[f]] + (uint64_t)cf->cost_us_per_token * (L - h[f]);
            all_over &= ttft[(size_t)r * d + f] > cf->slo_us;
            if (h[f] == hmax) {
                nmax++;
                if (a == d || s->W[c[f]] < s->W[c[a]]) a = f;
            }
        }
        uint32_t pick = a;
        const int over = nmax < d && ttft[(size_t)r * d + a] > cf->slo_us;
        if (over)
            for (uint32_t f = 0; f < d; f++)
                if (s->W[c[f]] < s->W[c[pick]]) pick = f;
        switched[r] = (uint8_t)over;
        const uint32_t ch = c[pick], hch = h[pick];
        chosen[r] = ch;
        if (all_over) s->both_over = 1;
        q_entry e;
        e.seq = s->next_seq++;
        e.L = L; e.c1 = c[0]; e.c2 = d > 1 ? c[1] : c[0]; e.h1 = h[0]; e.h2 = d > 1 ? h[1] : h[0];
        e.work = e.remaining = (uint64_t)cf->cost_us_per_token * (L - hch);
        e.moved_in_call = 0;
        e.arrival = t_batch;
        e.keys = NULL;
        e.nblk = s->pend_nblk[r];
        if ((cf->rebalance_flags & OR_RB_FRESH_HITS) && e.nblk) {
            e.keys = (uint64_t *)malloc((size_t)e.nblk * sizeof(uint64_t));
            if (!e.keys) return OR_ERR_OOM;
            memcpy(e.keys, s->pend_keys[r], (size_t)e.nblk * sizeof(uint64_t));
        }
        if (q_push(&s->q[ch], &e)) { free(e.keys); return OR_ERR_OOM; }
        s->W[ch] += e.work;
        s->pend_final[r] = ch;
        s->m_requests++;
        s->m_prompt_tokens += L;
        s->m_hit_tokens += hch;
        s->m_switched += switched[r];
        s->m_est_slo_met += s->W[ch] <= cf->slo_us;
    }
    if (n > 0) {
        s->m_cv_last = load_cv(s);
        s->m_cv_sum += s->m_cv_last;
        s->m_batches++;
    }
    s->pending = 1;
    return OR_OK;
}

int or_commit(or_state *s)
{
    if (!s->pending) return OR_OK;
    for (uint32_t r = 0; r < s->pend_n; r++) {
        lru_t *c = &s->cache[s->pend_final[r]];
        const uint64_t *keys = s->pend_keys[r];
        for (uint32_t b = s->pend_nblk[r]; b-- > 0;) {
            int rc = lru_touch(c, keys[b], ++s->clock, s->cfg.cache_capacity_blocks);
            if (rc) return rc;
        }
    }
    clear_pending(s);
    return OR_OK;
}

/* ------------------------------------------------------------------ */
/* Hotspot-aware rebalancing (Sec. 3.3)                                 */
/* ------------------------------------------------------------------ */

typedef struct {
    int64_t benefit;
    uint64_t seq;
    uint64_t ttft_i;
} mig_cand;

static int mig_cmp(const void *a, const void *b)
{
    const mig_cand *x = (const mig_cand *)a, *y = (const mig_cand *)b;
    if (x->benefit != y->benefit) return x->benefit > y->benefit ? -1 : 1;
    if (x->seq != y->seq) return x->seq < y->seq ? -1 : 1;
    return 0;
}

static int is_hot(const or_state *s, uint32_t i, uint64_t sumW, uint32_t N)
{
    /* hot_den * N * W_i > hot_num * sum(W), in 128-bit-safe form */
    unsigned __int128 lhs = (unsigned __int128)s->cfg.hot_den * N * s->W[i];
    unsigned __int128 rhs = (unsigned __int128)s->cfg.hot_num * sumW;
    return lhs > rhs;
}

/* Hit tokens of queue entry e on its candidate j: probed afresh against j's
 * cache with OR_RB_FRESH_HITS (when the entry kept its keys), else the hit
 * stored when it was routed. */
static uint32_t other_hit(const or_state *s, const q_entry *e, uint32_t j)
{
    if ((s->cfg.rebalance_flags & OR_RB_FRESH_HITS) && e->keys)
        return s->cfg.block_tokens * leading_hits(&s->cache[j], e->keys, e->nblk);
    return j == e->c1 ? e->h1 : e->h2;
}

int or_rebalance(or_state *s, uint64_t *mig_seq, uint32_t *mig_from, uint32_t *mig_to,
                 uint32_t cap, uint32_t *n_out)
{
    const or_config *cf = &s->cfg;
    const uint32_t M = cf->max_instances;
    uint64_t call = ++s->rebalance_calls;
    uint32_t nmig = 0;
    uint32_t N = n_live(s);
    uint64_t sumW = 0;
    for (uint32_t i = 0; i < M; i++) if (s->state[i] == INST_LIVE) sumW += s->W[i];
    const int slo_target = (cf->rebalance_flags & OR_RB_SLO_TARGET) != 0;
    *n_out = 0;
    if ((cf->rebalance_flags & OR_RB_DOUBLE_OVERLOAD) && !s->both_over) return OR_OK;

    /* hotspots at the start of the call, by W descending, then id */
    uint32_t *hot = (uint32_t *)malloc(M * sizeof(uint32_t));
    if (!hot) return OR_ERR_OOM;
    uint32_t nh = 0;
    for (uint32_t i = 0; i < M; i++)
        if (s->state[i] == INST_LIVE && (slo_target ? s->W[i] > cf->slo_us : is_hot(s, i, sumW, N)))
            hot[nh++] = i;
    for (uint32_t a = 1; a < nh; a++) {      /* insertion sort, stable by id */
        uint32_t x = hot[a], b = a;
        while (b > 0 && s->W[hot[b - 1]] < s->W[x]) { hot[b] = hot[b - 1]; b--; }
        hot[b] = x;
    }

    for (uint32_t hi = 0; hi < nh; hi++) {
        uint32_t i = hot[hi];
        queue_t *q = &s->q[i];
        mig_cand *cand = (mig_cand *)malloc((q->len ? q->len : 1) * sizeof(mig_cand));
        if (!cand) { free(hot); return OR_ERR_OOM; }
        uint32_t nc = 0;
        uint64_t ahead = 0;
        for (uint64_t k = 0; k < q->len; k++) {
            const q_entry *e = &q->e[q->head + k];
            uint64_t ttft_i = ahead + e->remaining;   /* T_q + T_c on i */
            ahead += e->remaining;
            if (e->remaining != e->work || e->moved_in_call == call) continue;
            uint32_t j = e->c1 == i ? e->c2 : e->c1;
            uint32_t hj = other_hit(s, e, j);
            uint64_t ttft_j = s->W[j] + (uint64_t)cf->cost_us_per_token * (e->L - hj);
            cand[nc].benefit = (int64_t)(ttft_i - ttft_j);
            cand[nc].seq = e->seq;
            cand[nc].ttft_i = ttft_i;
            nc++;
        }
        qsort(cand, nc, sizeof(mig_cand), mig_cmp);
        for (uint32_t a = 0; a < nc; a++) {
            if (slo_target ? !(s->W[i] > cf->slo_us) : !is_hot(s, i, sumW, N)) break;
            /* find the entry again (its position may have shifted) */
            uint64_t k = 0;
            while (k < q->len && q->e[q->head + k].seq != cand[a].seq) k++;
            q_entry e = q->e[q->head + k];
            uint32_t j = e.c1 == i ? e.c2 : e.c1;
            if (s->state[j] != INST_LIVE) continue;
            uint32_t hj = other_hit(s, &e, j);
            uint64_t new_work = (uint64_t)cf->cost_us_per_token * (e.L - hj);
            uint64_t ttft_j = s->W[j] + new_work;
            if (!(cand[a].ttft_i > ttft_j && ttft_j < cf->slo_us)) continue;
            q_erase(q, k);
            s->W[i] -= e.work;
            sumW -= e.work;
            e.work = e.remaining = new_work;
            e.moved_in_call = call;
            if (q_push(&s->q[j], &e)) { free(cand); free(hot); return OR_ERR_OOM; }
            s->W[j] += new_work;
            sumW += new_work;
            if (s->pending && e.seq >= s->pend_seq0 && e.seq < s->pend_seq0 + s->pend_n)
                s->pend_final[e.seq - s->pend_seq0] = j;
            if (nmig < cap) {
                mig_seq[nmig] = e.seq;
                mig_from[nmig] = i;
                mig_to[nmig] = j;
            }
            nmig++;
        }
        free(cand);
    }
    free(hot);
    *n_out = nmig;
    return OR_OK;
}

/* ------------------------------------------------------------------ */
/* Introspection (tests)                                               */
/* ------------------------------------------------------------------ */

void or_get_loads(const or_state *s, uint64_t *W) { memcpy(W, s->W, s->cfg.max_instances * sizeof(uint64_t)); }

void or_get_state(const or_state *s, uint8_t *st) { memcpy(st, s->state, s->cfg.max_instances); }

uint64_t or_clock(const or_state *s) { return s->clock; }

void or_key_material(const or_state *s, uint32_t *K1, uint32_t *K2, uint64_t *scalars)
{
    memcpy(K1, s->K1, s->cfg.block_tokens * sizeof(uint32_t));
    memcpy(K2, s->K2, s->cfg.block_tokens * sizeof(uint32_t));
    uint64_t v[7] = {s->G1, s->G2, s->Sc, s->Sr1, s->Sr2, s->Sv1, s->Sv2};
    memcpy(scalars, v, sizeof v);
}

/* Keys and route positions of one prompt under this state's key material. */
uint32_t or_prompt_keys(const or_state *s, const uint32_t *tok, uint32_t L, uint64_t *keys, uint64_t *pos)
{
    pos[0] = pos[1] = 0;
    if (L < s->cfg.block_tokens) return 0;
    return prompt_keys(s, tok, L, keys, pos);
}

/* Raw ring owners of positions (before the distinct fix). */
void or_ring_owners(const or_state *s, const uint64_t *pos, uint32_t n, int f, uint32_t *owner)
{
    if (f < 0 || (uint32_t)f >= s->nrings) return;
    for (uint32_t i = 0; i < n; i++) owner[i] = ring_owner(s, f, pos[i]);
}

/* Key material of function f (0-based): its NH keys (B words), and
 * scalars = {G, S_r, S_v}. */
void or_key_material_f(const or_state *s, uint32_t f, uint32_t *K, uint64_t *scalars)
{
    if (f >= s->nrings) return;
    const uint32_t *Kf = f == 0 ? s->K1 : f == 1 ? s->K2 : s->Kx[f - 2];
    memcpy(K, Kf, s->cfg.block_tokens * sizeof(uint32_t));
    scalars[0] = f == 0 ? s->G1 : f == 1 ? s->G2 : s->Gx[f - 2];
    scalars[1] = f == 0 ? s->Sr1 : f == 1 ? s->Sr2 : s->Srx[f - 2];
    scalars[2] = f == 0 ? s->Sv1 : f == 1 ? s->Sv2 : s->Svx[f - 2];
}

/* Ring position of a prompt under function f (0-based), hashed over its
 * first min(K_route, n_blk) blocks. */
uint64_t or_ring_position(const or_state *s, const uint32_t *tok, uint32_t L, uint32_t f)
{
    const uint32_t nblk = L / s->cfg.block_tokens;
    const uint32_t K = s->cfg.route_prefix_blocks < nblk ? s->cfg.route_prefix_blocks : nblk;
    return f < s->nrings ? ring_pos_f(s, tok, K, f) : 0;
}

uint32_t or_ring_dump(const or_state *s, int f, uint64_t *vpos, uint32_t *owner, uint32_t *vidx)
{
    if (f < 0 || (uint32_t)f >= s->nrings) return 0;
    for (uint32_t k = 0; k < s->ring_len; k++) {
        if (vpos) vpos[k] = s->ring[f][k].pos;
        if (owner) owner[k] = s->ring[f][k].id;
        if (vidx) vidx[k] = s->ring[f][k].v;
    }
    return s->ring_len;
}

uint32_t or_next_live(const or_state *s, uint32_t id) { return next_live_after(s, id); }

/* Resident keys of an instance, most recent first. */
uint64_t or_cache_dump(const or_state *s, uint32_t id, uint64_t *keys, uint64_t *stamps, uint64_t cap)
{
    const lru_t *c = &s->cache[id];
    uint64_t k = 0;
    for (int64_t i = c->mru; i >= 0; i = c->nodes[i].older, k++)
        if (k < cap) { keys[k] = c->nodes[i].key; stamps[k] = c->nodes[i].stamp; }
    return c->size;
}

/* Queue of an instance, head first: seq, work, remaining per entry. */
uint64_t or_queue_dump(const or_state *s, uint32_t id, uint64_t *seq, uint64_t *work,
                       uint64_t *remaining, uint64_t cap)
{
    const queue_t *q = &s->q[id];
    for (uint64_t k = 0; k < q->len && k < cap; k++) {
        seq[k] = q->e[q->head + k].seq;
        work[k] = q->e[q->head + k].work;
        remaining[k] = q->e[q->head + k].remaining;
    }
    return q->len;
}

/* Append a hand-built entry to an instance's queue (test set-up). */
int or_debug_enqueue(or_state *s, uint32_t id, uint64_t seq, uint32_t L, uint32_t c1, uint32_t c2,
                     uint32_t h1, uint32_t h2, uint64_t work, uint64_t remaining)
{
    if (id >= s->cfg.max_instances) return OR_ERR_INVALID_ARG;
    q_entry e = {seq, L, c1, c2, h1, h2, work, remaining, 0, s->t_prev, NULL, 0};
    int rc = q_push(&s->q[id], &e);
    if (!rc) s->W[id] += remaining;
    if (seq >= s->next_seq) s->next_seq = seq + 1;
    return rc;
}

/* Touch one key on one instance's LRU (test set-up of cache contents). */
int or_debug_touch(or_state *s, uint32_t id, uint64_t key)
{
    if (id >= s->cfg.max_instances) return OR_ERR_INVALID_ARG;
    return lru_touch(&s->cache[id], key, ++s->clock, s->cfg.cache_capacity_blocks);
}

/* ------------------------------------------------------------------ */
/* Metrics                                                             */
/* ------------------------------------------------------------------ */

/* Lower edge of the bucket holding the ceil(pnum/pden * count)-th smallest
 * value (rank at least 1); 0 when the histogram is empty. */
static uint64_t hist_percentile(const uint64_t *hist, uint64_t count, uint64_t pnum, uint64_t pden)
{
    if (count == 0) return 0;
    uint64_t rank = (pnum * count + pden - 1) / pden;
    if (rank == 0) rank = 1;
    uint64_t cum = 0;
    for (uint32_t k = 0; k < OR_HIST_BUCKETS; k++) {
        cum += hist[k];
        if (cum >= rank) return or_hist_lower(k);
    }
    return or_hist_lower(OR_HIST_BUCKETS - 1);
}

/* Metrics since create or the last reset.  u[0..12]: requests routed,
 * prompt tokens, hit tokens on the chosen candidates, switched, estimated
 * TTFT <= SLO, completed, TTFT sum, TTFT max, completed with TTFT <= SLO,
 * TTFT p50, p90, p99 (histogram lower edges), CV samples.  d[0..1]: sum of
 * the CV samples, the last one.  hist: OR_HIST_BUCKETS counts, or NULL. */
void or_get_metrics(or_state *s, uint64_t *u, double *d, uint64_t *hist, int reset)
{
    u[0] = s->m_requests; u[1] = s->m_prompt_tokens; u[2] = s->m_hit_tokens;
    u[3] = s->m_switched; u[4] = s->m_est_slo_met; u[5] = s->m_completed;
    u[6] = s->m_ttft_sum; u[7] = s->m_ttft_max; u[8] = s->m_slo_met;
    u[9] = hist_percentile(s->m_hist, s->m_completed, 50, 100);
    u[10] = hist_percentile(s->m_hist, s->m_completed, 90, 100);
    u[11] = hist_percentile(s->m_hist, s->m_completed, 99, 100);
    u[12] = s->m_batches;
    d[0] = s->m_cv_sum;
    d[1] = s->m_cv_last;
    if (hist) memcpy(hist, s->m_hist, sizeof s->m_hist);
    if (reset) {
        s->m_requests = s->m_prompt_tokens = s->m_hit_tokens = s->m_switched = 0;
        s->m_est_slo_met = s->m_completed = s->m_ttft_sum = s->m_ttft_max = 0;
        s->m_slo_met = s->m_batches = 0;
        s->m_cv_sum = s->m_cv_last = 0.0;
        memset(s->m_hist, 0, sizeof s->m_hist);
    }
}

/* Hash prefix length (blocks) of each request of the last routed batch;
 * returns the batch size. */
uint32_t or_last_route_blocks(const or_state *s, uint32_t *K)
{
    if (K && s->last_n) memcpy(K, s->last_K, s->last_n * sizeof(uint32_t));
    return s->last_n;
}

/* Expanded nodes of the prefix hotness tree (sorted keys); returns their
 * number (entries beyond cap are not written). */
uint64_t or_prefix_tree(const or_state *s, uint64_t *keys, uint64_t cap)
{
    for (uint64_t i = 0; i < s->ad_set_n && i < cap; i++) keys[i] = s->ad_set[i];
    return s->ad_set_n;
}

/* ------------------------------------------------------------------ */
/* Power of d choices (App. A.8, "Optimal Candidate Set Size")          */
/* ------------------------------------------------------------------ */

/* Choice k of ball t in trial s: with c = (s * m + t) * d + k, the value
 * x_c = the (c+1)-th output of SplitMix64 seeded with `seed`, and the bin
 * floor(x_c * n / 2^64). */
uint32_t or_potc_choice(uint64_t seed, uint64_t c, uint32_t n)
{
    uint64_t state = seed + c * 0x9E3779B97F4A7C15ULL;   /* the state before output c+1 */
    uint64_t x = or_splitmix64_next(&state);
    return (uint32_t)(((unsigned __int128)x * n) >> 64);
}

/* Place one ball: the least loaded of its d choices, ties to the earlier
 * choice. */
static uint32_t potc_place(uint32_t *load, const uint32_t *choice, uint32_t d)
{
    uint32_t best = choice[0];
    for (uint32_t k = 1; k < d; k++)
        if (load[choice[k]] < load[best]) best = choice[k];
    load[best]++;
    return best;
}

/* Hand-given choices (tests): choices[t*d + k]; fills load[n]. */
void or_potc_place_all(const uint32_t *choices, uint64_t m, uint32_t d, uint32_t n, uint32_t *load)
{
    memset(load, 0, n * sizeof(uint32_t));
    for (uint64_t t = 0; t < m; t++) potc_place(load, choices + t * d, d);
}

/* Maximum bin load of each of `trials` trials of m balls into n bins with
 * d choices each. */
int or_potc_max_loads(uint32_t n, uint64_t m, uint32_t d, uint32_t trials, uint64_t seed, uint32_t *max_load)
{
    if (n < 1 || d < 1 || d > 64) return OR_ERR_INVALID_ARG;
    uint32_t *load = (uint32_t *)malloc(n * sizeof(uint32_t));
    if (!load) return OR_ERR_OOM;
    uint32_t choice[64];
    for (uint32_t s = 0; s < trials; s++) {
        memset(load, 0, n * sizeof(uint32_t));
        for (uint64_t t = 0; t < m; t++) {
            for (uint32_t k = 0; k < d; k++) choice[k] = or_potc_choice(seed, ((uint64_t)s * m + t) * d + k, n);
            potc_place(load, choice, d);
        }
        uint32_t mx = 0;
        for (uint32_t i = 0; i < n; i++) if (load[i] > mx) mx = load[i];
        max_load[s] = mx;
    }
    free(load);
    return OR_OK;
}
