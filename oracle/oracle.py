"""ctypes wrapper of the plain-C DualMap oracle (dm_oracle.c).

TEST INFRASTRUCTURE ONLY: the test-suite, the smoke check and the CPU-baseline
leg of the benchmark may import this module; the product path never does.
"""

import ctypes as C
import os
import subprocess

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "dm_oracle.c")
LIB = os.path.join(HERE, "liboracle_dm.so")

OK, ERR_INVALID_ARG, ERR_CAPACITY, ERR_NO_INSTANCES = 0, 1, 2, 3
ERR_DUPLICATE_ID, ERR_UNKNOWN_ID, ERR_ORDER = 4, 5, 6


def build(force=False):
    """Compile the oracle with the host C compiler (plain C, -O2)."""
    if not force and os.path.exists(LIB) and os.path.getmtime(LIB) >= os.path.getmtime(SRC):
        return LIB
    tmp = LIB + f".tmp{os.getpid()}"
    subprocess.check_call(["gcc", "-O2", "-std=gnu11", "-shared", "-fPIC", "-Wall", "-Wextra",
                           "-Wno-unused-parameter", SRC, "-o", tmp, "-lm"])
    os.replace(tmp, LIB)
    return LIB


class or_config(C.Structure):
    _fields_ = [
        ("block_tokens", C.c_uint32),
        ("route_prefix_blocks", C.c_uint32),
        ("vnodes_per_instance", C.c_uint32),
        ("max_instances", C.c_uint32),
        ("cache_capacity_blocks", C.c_uint64),
        ("slo_us", C.c_uint64),
        ("cost_us_per_token", C.c_uint32),
        ("hot_num", C.c_uint32),
        ("hot_den", C.c_uint32),
        ("max_batch", C.c_uint32),
        ("max_batch_tokens", C.c_uint64),
        ("seed", C.c_uint64),
        ("choice_rule", C.c_uint32),
        ("adapt_step_blocks", C.c_uint32),
        ("adapt_max_blocks", C.c_uint32),
        ("adapt_window", C.c_uint32),
        ("rebalance_flags", C.c_uint32),
        ("candidates", C.c_uint32),
    ]


RULE_DUALMAP, RULE_CACHE_AFFINITY, RULE_LEAST_LOADED, RULE_MIN_TTFT, RULE_PREBLE = 0, 1, 2, 3, 4
RULE_GLOBAL_CACHE_AFFINITY, RULE_GLOBAL_LEAST_LOADED, RULE_GLOBAL_MIN_TTFT, RULE_GLOBAL_PREBLE = 5, 6, 7, 8
HIST_BUCKETS = 976
RB_SLO_TARGET, RB_DOUBLE_OVERLOAD, RB_FRESH_HITS = 1, 2, 4
METRIC_KEYS = ["requests", "prompt_tokens", "hit_tokens", "switched", "est_slo_met", "completed",
               "ttft_sum_us", "ttft_max_us", "slo_met", "ttft_p50_us", "ttft_p90_us", "ttft_p99_us",
               "cv_samples"]


_lib = None
u32p = np.ctypeslib.ndpointer(np.uint32, flags="C_CONTIGUOUS")
u64p = np.ctypeslib.ndpointer(np.uint64, flags="C_CONTIGUOUS")
u8p = np.ctypeslib.ndpointer(np.uint8, flags="C_CONTIGUOUS")


def lib():
    global _lib
    if _lib is None:
        build()
        L = C.CDLL(LIB)
        V, P = C.c_void_p, C.POINTER
        sig = {
            "or_splitmix64_next": (C.c_uint64, [P(C.c_uint64)]),
            "or_mix64": (C.c_uint64, [C.c_uint64]),
            "or_fmix64": (C.c_uint64, [C.c_uint64]),
            "or_nh": (C.c_uint64, [u32p, u32p, C.c_uint32]),
            "or_derive_keys": (None, [C.c_uint64, C.c_uint32, u32p, u32p, u64p]),
            "or_vnode_pos": (C.c_uint64, [C.c_uint64, C.c_uint32, C.c_uint32]),
            "or_ring_successor": (C.c_uint32, [u64p, C.c_uint32, C.c_uint64]),
            "or_create": (C.c_int, [P(or_config), P(V)]),
            "or_destroy": (None, [V]),
            "or_add_instance": (C.c_int, [V, C.c_uint32]),
            "or_remove_instance": (C.c_int, [V, C.c_uint32]),
            "or_choose": (C.c_uint32, [C.c_uint32, C.c_uint32, C.c_uint32, C.c_uint32, C.c_uint32, C.c_uint32,
                                       C.c_uint64, C.c_uint64, C.c_uint64, C.c_uint32,
                                       P(C.c_uint64), P(C.c_uint64), P(C.c_uint8)]),
            "or_route_part": (C.c_int, [V, u32p, u64p, u32p, C.c_uint32, C.c_uint32, u32p, u32p, u32p, u32p,
                                        u32p, u64p, C.c_uint64]),
            "or_route_given": (C.c_int, [V, u32p, C.c_uint32, C.c_uint64, u32p, u32p, u32p, u32p, u32p, u64p,
                                         u64p, u64p, u32p, u8p]),
            "or_route_batch": (C.c_int, [V, u32p, u64p, u32p, C.c_uint32, C.c_uint64,
                                         u32p, u32p, u32p, u32p, u64p, u64p, u32p, u8p]),
            "or_commit": (C.c_int, [V]),
            "or_rebalance": (C.c_int, [V, u64p, u32p, u32p, C.c_uint32, P(C.c_uint32)]),
            "or_get_loads": (None, [V, u64p]),
            "or_get_state": (None, [V, u8p]),
            "or_clock": (C.c_uint64, [V]),
            "or_key_material": (None, [V, u32p, u32p, u64p]),
            "or_prompt_keys": (C.c_uint32, [V, u32p, C.c_uint32, u64p, u64p]),
            "or_ring_owners": (None, [V, u64p, C.c_uint32, C.c_int, u32p]),
            "or_ring_dump": (C.c_uint32, [V, C.c_int, V, V, V]),
            "or_next_live": (C.c_uint32, [V, C.c_uint32]),
            "or_cache_dump": (C.c_uint64, [V, C.c_uint32, u64p, u64p, C.c_uint64]),
            "or_queue_dump": (C.c_uint64, [V, C.c_uint32, u64p, u64p, u64p, C.c_uint64]),
            "or_debug_enqueue": (C.c_int, [V, C.c_uint32, C.c_uint64, C.c_uint32, C.c_uint32,
                                           C.c_uint32, C.c_uint32, C.c_uint32, C.c_uint64,
                                           C.c_uint64]),
            "or_debug_touch": (C.c_int, [V, C.c_uint32, C.c_uint64]),
            "or_hist_bucket": (C.c_uint32, [C.c_uint64]),
            "or_hist_lower": (C.c_uint64, [C.c_uint32]),
            "or_get_metrics": (None, [V, u64p, P(C.c_double), V, C.c_int]),
            "or_last_route_blocks": (C.c_uint32, [V, V]),
            "or_potc_choice": (C.c_uint32, [C.c_uint64, C.c_uint64, C.c_uint32]),
            "or_potc_place_all": (None, [u32p, C.c_uint64, C.c_uint32, C.c_uint32, u32p]),
            "or_potc_max_loads": (C.c_int, [C.c_uint32, C.c_uint64, C.c_uint32, C.c_uint32, C.c_uint64, u32p]),
            "or_prefix_tree": (C.c_uint64, [V, V, C.c_uint64]),
            "or_route_batch_d": (C.c_int, [V, C.c_uint32, u32p, u64p, u32p, C.c_uint32, C.c_uint64,
                                           u32p, u32p, u64p, u32p, u8p]),
            "or_ring_position": (C.c_uint64, [V, u32p, C.c_uint32, C.c_uint32]),
            "or_key_material_f": (None, [V, C.c_uint32, u32p, u64p]),
        }
        for name, (res, args) in sig.items():
            f = getattr(L, name)
            f.restype = res
            f.argtypes = args
        _lib = L
    return _lib


# -- primitives -------------------------------------------------------------

def splitmix64_stream(seed, n):
    s = C.c_uint64(seed)
    return [lib().or_splitmix64_next(C.byref(s)) for _ in range(n)]


def mix64(x):
    return lib().or_mix64(x)


def fmix64(x):
    return lib().or_fmix64(x)


def nh(tokens, key):
    t = np.ascontiguousarray(tokens, dtype=np.uint32)
    k = np.ascontiguousarray(key, dtype=np.uint32)
    return lib().or_nh(t, k, len(t))


def derive_keys(seed, B):
    K1 = np.zeros(B, np.uint32)
    K2 = np.zeros(B, np.uint32)
    sc = np.zeros(7, np.uint64)
    lib().or_derive_keys(seed, B, K1, K2, sc)
    return K1, K2, sc


def vnode_pos(Sv, id_, v):
    return lib().or_vnode_pos(Sv, id_, v)


def ring_successor(vpos, p):
    vp = np.ascontiguousarray(vpos, dtype=np.uint64)
    return lib().or_ring_successor(vp, len(vp), p)


def choose(c1, c2, h1, h2, L, W1, W2, slo, cost=1, rule=RULE_DUALMAP):
    t1, t2, sw = C.c_uint64(), C.c_uint64(), C.c_uint8()
    ch = lib().or_choose(rule, c1, c2, h1, h2, L, W1, W2, slo, cost, C.byref(t1), C.byref(t2),
                         C.byref(sw))
    return ch, t1.value, t2.value, sw.value


def potc_choice(seed, c, n):
    return lib().or_potc_choice(seed, c, n)


def potc_place_all(choices, n):
    ch = np.ascontiguousarray(choices, dtype=np.uint32)
    load = np.zeros(n, np.uint32)
    lib().or_potc_place_all(ch.reshape(-1), ch.shape[0], ch.shape[1], n, load)
    return load


def potc_max_loads(n, m, d, trials, seed):
    out = np.zeros(max(trials, 1), np.uint32)
    rc = lib().or_potc_max_loads(n, m, d, trials, seed, out)
    if rc:
        raise ValueError(f"or_potc_max_loads: {rc}")
    return out[:trials]


def hist_bucket(v):
    return lib().or_hist_bucket(v)


def hist_lower(k):
    return lib().or_hist_lower(k)


def config_from_workload(w, **kw):
    """Oracle config for a workload dict (tracegen.configs)."""
    d = dict(block_tokens=w["block_tokens"], route_prefix_blocks=w["route_prefix_blocks"],
             vnodes_per_instance=w["vnodes"], max_instances=kw.pop("max_instances", w["n_instances"] + 16),
             cache_capacity_blocks=w["capacity"], slo_us=w["slo_us"], cost_us_per_token=w["cost_us"],
             hot_num=3, hot_den=2, max_batch=w["batch"], max_batch_tokens=kw.pop("max_batch_tokens", 1 << 40),
             seed=w["seed"])
    d.update(kw)
    return d


class Oracle:
    """One oracle scheduler state."""

    def __init__(self, **cfg):
        self.cfg = or_config(**cfg)
        h = C.c_void_p()
        rc = lib().or_create(C.byref(self.cfg), C.byref(h))
        if rc:
            raise ValueError(f"or_create failed: {rc}")
        self.h = h
        self.M = self.cfg.max_instances
        self.B = self.cfg.block_tokens

    def __del__(self):
        if getattr(self, "h", None):
            lib().or_destroy(self.h)
            self.h = None

    def add_instance(self, i):
        return lib().or_add_instance(self.h, i)

    def remove_instance(self, i):
        return lib().or_remove_instance(self.h, i)

    def route_batch(self, tokens, offsets, lengths, t_batch):
        n = len(lengths)
        out = dict(cand1=np.zeros(n, np.uint32), cand2=np.zeros(n, np.uint32),
                   hit1=np.zeros(n, np.uint32), hit2=np.zeros(n, np.uint32),
                   ttft1=np.zeros(n, np.uint64), ttft2=np.zeros(n, np.uint64),
                   chosen=np.zeros(n, np.uint32), switched=np.zeros(n, np.uint8))
        tok = np.ascontiguousarray(tokens, dtype=np.uint32)
        if tok.size == 0:
            tok = np.zeros(1, np.uint32)
        rc = lib().or_route_batch(self.h, tok, np.ascontiguousarray(offsets, dtype=np.uint64),
                                  np.ascontiguousarray(lengths, dtype=np.uint32), n, t_batch,
                                  out["cand1"], out["cand2"], out["hit1"], out["hit2"],
                                  out["ttft1"], out["ttft2"], out["chosen"], out["switched"])
        return rc, out

    def route_part(self, tokens, offsets, lengths, r0, r1):
        """Sharded routing, one rank's half: keys (concatenated), hash length,
        candidates and hits of requests r0 .. r1-1, the state unchanged."""
        B = self.B
        lens = np.ascontiguousarray(lengths, dtype=np.uint32)
        k = r1 - r0
        out = dict(K=np.zeros(k, np.uint32), cand1=np.zeros(k, np.uint32), cand2=np.zeros(k, np.uint32),
                   hit1=np.zeros(k, np.uint32), hit2=np.zeros(k, np.uint32))
        cap = int((lens[r0:r1] // B).sum())
        keys = np.zeros(max(cap, 1), np.uint64)
        tok = np.ascontiguousarray(tokens, dtype=np.uint32)
        if tok.size == 0:
            tok = np.zeros(1, np.uint32)
        rc = lib().or_route_part(self.h, tok, np.ascontiguousarray(offsets, dtype=np.uint64), lens, r0, r1,
                                 out["K"], out["cand1"], out["cand2"], out["hit1"], out["hit2"], keys, cap)
        out["keys"] = keys[:cap]
        return rc, out

    def route_given(self, lengths, t_batch, K, cand1, cand2, hit1, hit2, keys):
        """Sharded routing, the replicated half: the batch routed with every
        request's keys, hash length, candidates and hits given."""
        lens = np.ascontiguousarray(lengths, dtype=np.uint32)
        n = len(lens)
        out = dict(ttft1=np.zeros(n, np.uint64), ttft2=np.zeros(n, np.uint64), chosen=np.zeros(n, np.uint32),
                   switched=np.zeros(n, np.uint8))
        a = lambda x, t: np.ascontiguousarray(x, dtype=t)
        kk = a(keys, np.uint64)
        if kk.size == 0:
            kk = np.zeros(1, np.uint64)
        rc = lib().or_route_given(self.h, lens, n, t_batch, a(K, np.uint32), a(cand1, np.uint32),
                                  a(cand2, np.uint32), a(hit1, np.uint32), a(hit2, np.uint32), kk,
                                  out["ttft1"], out["ttft2"], out["chosen"], out["switched"])
        return rc, out

    def route_batch_d(self, d, tokens, offsets, lengths, t_batch):
        """Routing with d candidates (App. A.8): (status, dict of cand, hit,
        ttft as n x d arrays, chosen and switched)."""
        n = len(lengths)
        cand = np.zeros(n * d, np.uint32)
        hit = np.zeros(n * d, np.uint32)
        ttft = np.zeros(n * d, np.uint64)
        chosen = np.zeros(n, np.uint32)
        sw = np.zeros(n, np.uint8)
        tok = np.ascontiguousarray(tokens, dtype=np.uint32)
        rc = lib().or_route_batch_d(self.h, d, tok if tok.size else np.zeros(1, np.uint32),
                                    np.ascontiguousarray(offsets, dtype=np.uint64),
                                    np.ascontiguousarray(lengths, dtype=np.uint32), n, t_batch, cand, hit, ttft,
                                    chosen, sw)
        return rc, dict(cand=cand.reshape(n, d), hit=hit.reshape(n, d), ttft=ttft.reshape(n, d), chosen=chosen,
                        switched=sw)

    def ring_position(self, tokens, f):
        t = np.ascontiguousarray(tokens, dtype=np.uint32)
        return lib().or_ring_position(self.h, t, len(t), f)

    def key_material_f(self, f):
        K = np.zeros(self.B, np.uint32)
        sc = np.zeros(3, np.uint64)
        lib().or_key_material_f(self.h, f, K, sc)
        return K, sc

    def commit(self):
        return lib().or_commit(self.h)

    def route_blocks(self):
        """Hash prefix length (blocks) of each request of the last batch."""
        n = lib().or_last_route_blocks(self.h, None)
        K = np.zeros(max(n, 1), np.uint32)
        lib().or_last_route_blocks(self.h, K.ctypes.data)
        return K[:n]

    def prefix_tree(self):
        """Sorted keys of the expanded nodes of the prefix hotness tree."""
        n = lib().or_prefix_tree(self.h, None, 0)
        k = np.zeros(max(n, 1), np.uint64)
        lib().or_prefix_tree(self.h, k.ctypes.data, n)
        return k[:n]

    def metrics(self, reset=False):
        """Counters (METRIC_KEYS), cv_sum, cv_last and the TTFT histogram."""
        u = np.zeros(len(METRIC_KEYS), np.uint64)
        d = (C.c_double * 2)()
        hist = np.zeros(HIST_BUCKETS, np.uint64)
        lib().or_get_metrics(self.h, u, d, hist.ctypes.data, 1 if reset else 0)
        m = {k: int(v) for k, v in zip(METRIC_KEYS, u)}
        m["cv_sum"], m["cv_last"] = d[0], d[1]
        return m, hist

    def rebalance(self, cap=1 << 16):
        seq = np.zeros(cap, np.uint64)
        fr = np.zeros(cap, np.uint32)
        to = np.zeros(cap, np.uint32)
        n = C.c_uint32()
        rc = lib().or_rebalance(self.h, seq, fr, to, cap, C.byref(n))
        k = min(n.value, cap)
        return rc, n.value, (seq[:k], fr[:k], to[:k])

    def loads(self):
        W = np.zeros(self.M, np.uint64)
        lib().or_get_loads(self.h, W)
        return W

    def inst_state(self):
        st = np.zeros(self.M, np.uint8)
        lib().or_get_state(self.h, st)
        return st

    def clock(self):
        return lib().or_clock(self.h)

    def key_material(self):
        K1 = np.zeros(self.B, np.uint32)
        K2 = np.zeros(self.B, np.uint32)
        sc = np.zeros(7, np.uint64)
        lib().or_key_material(self.h, K1, K2, sc)
        return K1, K2, sc

    def prompt_keys(self, tokens):
        t = np.ascontiguousarray(tokens, dtype=np.uint32)
        keys = np.zeros(max(1, len(t) // self.B), np.uint64)
        pos = np.zeros(2, np.uint64)
        nb = lib().or_prompt_keys(self.h, t if t.size else np.zeros(1, np.uint32), len(t), keys, pos)
        return keys[:nb], pos

    def ring_owners(self, pos, f):
        p = np.ascontiguousarray(pos, dtype=np.uint64)
        o = np.zeros(len(p), np.uint32)
        lib().or_ring_owners(self.h, p, len(p), f, o)
        return o

    def ring(self, f):
        n = lib().or_ring_dump(self.h, f, None, None, None)
        vp = np.zeros(max(n, 1), np.uint64)
        ow = np.zeros(max(n, 1), np.uint32)
        vi = np.zeros(max(n, 1), np.uint32)
        lib().or_ring_dump(self.h, f, vp.ctypes.data, ow.ctypes.data, vi.ctypes.data)
        return vp[:n], ow[:n], vi[:n]

    def next_live(self, i):
        return lib().or_next_live(self.h, i)

    def cache(self, i, cap=None):
        n = lib().or_cache_dump(self.h, i, np.zeros(1, np.uint64), np.zeros(1, np.uint64), 0)
        cap = n if cap is None else cap
        k = np.zeros(max(cap, 1), np.uint64)
        s = np.zeros(max(cap, 1), np.uint64)
        lib().or_cache_dump(self.h, i, k, s, cap)
        m = min(n, cap)
        return k[:m], s[:m]

    def queue(self, i, cap=1 << 20):
        seq = np.zeros(cap, np.uint64)
        work = np.zeros(cap, np.uint64)
        rem = np.zeros(cap, np.uint64)
        n = lib().or_queue_dump(self.h, i, seq, work, rem, cap)
        m = min(n, cap)
        return seq[:m], work[:m], rem[:m]

    def debug_enqueue(self, i, seq, L, c1, c2, h1, h2, work, remaining=None):
        return lib().or_debug_enqueue(self.h, i, seq, L, c1, c2, h1, h2, work,
                                      work if remaining is None else remaining)

    def debug_touch(self, i, key):
        return lib().or_debug_touch(self.h, i, key)
