"""ctypes binding of libdualmap.so (include/dualmap.h).

Argument marshalling only: every step of the routing path runs in the
library's CUDA kernels.  PyTorch supplies device memory and streams.  There
is no fallback: if the shared library is missing, importing the binding's
functions raises.
"""

import ctypes as C
import os

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
# DM_LIBRARY=debug loads the debug build (bounds checks, DM_ERR_BOUNDS);
# it is made by build.build(debug=True).  Read once, at the first lib() call.
LIB_PATH = os.path.join(HERE, "libdualmap_debug.so" if os.environ.get("DM_LIBRARY") == "debug" else "libdualmap.so")

DM_OK, DM_ERR_INVALID_ARG, DM_ERR_CAPACITY, DM_ERR_NO_INSTANCES = 0, 1, 2, 3
DM_ERR_DUPLICATE_ID, DM_ERR_UNKNOWN_ID, DM_ERR_ORDER, DM_ERR_CUDA = 4, 5, 6, 7
DM_ERR_TIMEOUT, DM_ERR_OOM, DM_ERR_BOUNDS = 8, 9, 10
STAGES = ["setup", "drain", "hash", "probe", "choice", "commit", "rebalance"]

# dm_choice_rule
DM_RULE_DUALMAP, DM_RULE_PAIR_CACHE_AFFINITY, DM_RULE_PAIR_LEAST_LOADED = 0, 1, 2
DM_RULE_PAIR_MIN_TTFT, DM_RULE_PAIR_PREBLE = 3, 4
DM_RULE_CACHE_AFFINITY, DM_RULE_LEAST_LOADED, DM_RULE_MIN_TTFT, DM_RULE_PREBLE = 5, 6, 7, 8
RULE_NAMES = ["dualmap", "pair_cache_affinity", "pair_least_loaded", "pair_min_ttft", "pair_preble",
              "cache_affinity", "least_loaded", "min_ttft", "preble"]
DM_HIST_BUCKETS = 976
DM_REBALANCE_SLO_TARGET, DM_REBALANCE_DOUBLE_OVERLOAD, DM_REBALANCE_FRESH_HITS = 1, 2, 4


class dm_config(C.Structure):
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
        ("max_touch_per_instance", C.c_uint64),
        ("max_queue", C.c_uint32),
        ("index_slots_log2", C.c_uint32),
        ("choice_rule", C.c_uint32),
        ("adapt_step_blocks", C.c_uint32),
        ("adapt_max_blocks", C.c_uint32),
        ("adapt_window", C.c_uint32),
        ("rebalance_flags", C.c_uint32),
        ("rebuild_pool", C.c_uint32),
        ("test_loop_limit", C.c_uint32),
        ("candidates", C.c_uint32),
        ("rebalance_key_blocks", C.c_uint64),
        ("seed", C.c_uint64),
        ("stream", C.c_void_p),
    ]


class dm_batch(C.Structure):
    _fields_ = [
        ("tokens", C.c_void_p),
        ("offsets", C.c_void_p),
        ("lengths", C.c_void_p),
        ("n", C.c_uint32),
        ("reserved0", C.c_uint32),
        ("total_tokens", C.c_uint64),
        ("batch_time_us", C.c_uint64),
    ]


class dm_route_out(C.Structure):
    _fields_ = [(name, C.c_void_p) for name in
                ("cand1", "cand2", "hit1", "hit2", "ttft1", "ttft2", "chosen", "switched")]


class dm_route_out_d(C.Structure):
    _fields_ = [(name, C.c_void_p) for name in ("cand", "hit", "ttft", "chosen", "switched")]


class dm_metrics(C.Structure):
    _fields_ = [(name, C.c_uint64) for name in
                ("requests", "prompt_tokens", "hit_tokens", "switched", "est_slo_met", "completed", "ttft_sum_us",
                 "ttft_max_us", "slo_met", "ttft_p50_us", "ttft_p90_us", "ttft_p99_us", "cv_samples")] + \
               [("cv_sum", C.c_double), ("cv_last", C.c_double)]


class dm_migration(C.Structure):
    _fields_ = [("req_seq", C.c_uint64), ("from_", C.c_uint32), ("to", C.c_uint32)]


class DualMapError(RuntimeError):
    def __init__(self, status, where):
        self.status = status
        super().__init__(f"{where}: {status_string(status)} ({status})")


_lib = None

# name -> (restype, argtypes); the exported set is exactly include/dualmap.h
SIGNATURES = {
    "dm_create": (C.c_int, [C.POINTER(dm_config), C.POINTER(C.c_void_p)]),
    "dm_destroy": (None, [C.c_void_p]),
    "dm_add_instance": (C.c_int, [C.c_void_p, C.c_uint32]),
    "dm_remove_instance": (C.c_int, [C.c_void_p, C.c_uint32]),
    "dm_route_batch": (C.c_int, [C.c_void_p, C.POINTER(dm_batch), C.POINTER(dm_route_out)]),
    "dm_route_batch_host": (C.c_int, [C.c_void_p, C.POINTER(dm_batch), C.POINTER(dm_route_out)]),
    "dm_route_batch_d": (C.c_int, [C.c_void_p, C.POINTER(dm_batch), C.POINTER(dm_route_out_d)]),
    "dm_route_batch_host_async": (C.c_int, [C.c_void_p, C.POINTER(dm_batch), C.POINTER(dm_route_out)]),
    "dm_route_shard_begin": (C.c_int, [C.c_void_p, C.POINTER(dm_batch), C.c_uint32, C.c_uint32]),
    "dm_shard_export": (C.c_int, [C.c_void_p, C.c_uint32, C.c_uint32, C.c_void_p, C.c_uint64, C.c_void_p]),
    "dm_shard_import": (C.c_int, [C.c_void_p, C.c_uint32, C.c_uint32, C.c_void_p, C.c_uint64]),
    "dm_route_shard_finish": (C.c_int, [C.c_void_p, C.POINTER(dm_batch), C.POINTER(dm_route_out)]),
    "dm_rebalance": (C.c_int, [C.c_void_p, C.c_void_p, C.c_uint32, C.POINTER(C.c_uint32)]),
    "dm_rebalance_async": (C.c_int, [C.c_void_p, C.c_void_p, C.c_uint32, C.c_void_p]),
    "dm_commit_cache": (C.c_int, [C.c_void_p]),
    "dm_hash_prompts": (C.c_int, [C.c_void_p, C.POINTER(dm_batch), C.c_void_p, C.c_void_p, C.c_void_p]),
    "dm_hash_prompts_noalloc": (C.c_int, [C.c_uint32, C.c_uint32, C.c_uint64, C.POINTER(dm_batch), C.c_void_p,
                                          C.c_void_p, C.c_void_p, C.c_void_p]),
    "dm_ring_lookup": (C.c_int, [C.c_void_p, C.c_void_p, C.c_uint32, C.c_void_p, C.c_void_p]),
    "dm_get_loads": (C.c_int, [C.c_void_p, C.c_void_p, C.c_uint32, C.POINTER(C.c_uint32)]),
    "dm_export_cache": (C.c_int, [C.c_void_p, C.c_uint32, C.c_void_p, C.c_void_p, C.c_uint64,
                                  C.POINTER(C.c_uint64)]),
    "dm_export_queue": (C.c_int, [C.c_void_p, C.c_uint32, C.c_void_p, C.c_void_p, C.c_void_p, C.c_uint64,
                                  C.POINTER(C.c_uint64)]),
    "dm_export_ring": (C.c_int, [C.c_void_p, C.c_int, C.c_void_p, C.c_void_p, C.c_uint32,
                                 C.POINTER(C.c_uint32)]),
    "dm_get_clock": (C.c_int, [C.c_void_p, C.POINTER(C.c_uint64)]),
    "dm_get_maint_counts": (C.c_int, [C.c_void_p, C.POINTER(C.c_uint64), C.POINTER(C.c_uint64)]),
    "dm_get_metrics": (C.c_int, [C.c_void_p, C.POINTER(dm_metrics), C.c_void_p, C.c_uint32, C.c_int]),
    "dm_get_route_blocks": (C.c_int, [C.c_void_p, C.c_void_p, C.c_uint32]),
    "dm_export_prefix_tree": (C.c_int, [C.c_void_p, C.c_void_p, C.c_uint64, C.POINTER(C.c_uint64)]),
    "dm_potc_max_loads": (C.c_int, [C.c_uint32, C.c_uint64, C.c_uint32, C.c_uint32, C.c_uint64, C.c_void_p,
                                    C.c_void_p]),
    "dm_test_fail_alloc": (None, [C.c_int64]),
    "dm_last_error": (C.c_int, [C.c_void_p]),
    "dm_set_profiling": (C.c_int, [C.c_void_p, C.c_int]),
    "dm_get_stage_times": (C.c_int, [C.c_void_p, C.c_void_p, C.c_void_p, C.c_int]),
    "dm_status_string": (C.c_char_p, [C.c_int]),
}


def lib():
    """The loaded shared library; raises if it has not been built."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is missing: build it with "
                               "`python -c 'import __graft_entry__ as g; g.build()'`")
        L = C.CDLL(LIB_PATH)
        for name, (res, args) in SIGNATURES.items():
            f = getattr(L, name)
            f.restype = res
            f.argtypes = args
        _lib = L
    return _lib


def status_string(s):
    return lib().dm_status_string(s).decode()


def _check(rc, where):
    if rc != DM_OK:
        raise DualMapError(rc, where)


def _ptr(t):
    """Device (or host) address of a torch tensor / numpy array, or None."""
    if t is None:
        return None
    if hasattr(t, "data_ptr"):
        return t.data_ptr()
    return t.ctypes.data


# -- the C ABI, name for name ------------------------------------------------

def dm_create(cfg):
    h = C.c_void_p()
    _check(lib().dm_create(C.byref(cfg), C.byref(h)), "dm_create")
    return h


def dm_destroy(h):
    lib().dm_destroy(h)


def dm_add_instance(h, i):
    return lib().dm_add_instance(h, i)


def dm_remove_instance(h, i):
    return lib().dm_remove_instance(h, i)


def make_batch(tokens, offsets, lengths, n, total_tokens, batch_time_us):
    return dm_batch(_ptr(tokens), _ptr(offsets), _ptr(lengths), n, 0, total_tokens, batch_time_us)


def make_out(cand1, cand2, hit1, hit2, ttft1, ttft2, chosen, switched):
    return dm_route_out(*[_ptr(x) for x in (cand1, cand2, hit1, hit2, ttft1, ttft2, chosen, switched)])


def dm_route_batch(h, batch, out):
    return lib().dm_route_batch(h, C.byref(batch), C.byref(out))


def dm_route_batch_d(h, batch, out):
    return lib().dm_route_batch_d(h, C.byref(batch), C.byref(out))


def dm_route_shard_begin(h, batch, r0, r1):
    return lib().dm_route_shard_begin(h, C.byref(batch), r0, r1)


def dm_shard_export(h, r0, r1, buf_dev, cap, bytes_dev):
    return lib().dm_shard_export(h, r0, r1, _ptr(buf_dev), cap, _ptr(bytes_dev))


def dm_shard_import(h, r0, r1, buf_dev, nbytes):
    return lib().dm_shard_import(h, r0, r1, _ptr(buf_dev), nbytes)


def dm_route_shard_finish(h, batch, out):
    return lib().dm_route_shard_finish(h, C.byref(batch), C.byref(out))


def dm_route_batch_host(h, batch, out):
    return lib().dm_route_batch_host(h, C.byref(batch), C.byref(out))


def dm_route_batch_host_async(h, batch, out):
    return lib().dm_route_batch_host_async(h, C.byref(batch), C.byref(out))


def dm_rebalance(h, cap):
    """Synchronous rebalance with host results: (status, count, migrations
    as a numpy structured array of up to cap entries)."""
    out = (dm_migration * max(cap, 1))()
    n = C.c_uint32()
    rc = lib().dm_rebalance(h, out, cap, C.byref(n))
    m = np.ctypeslib.as_array(out)[:min(n.value, cap)] if rc == 0 else None
    return rc, n.value, m


def dm_rebalance_async(h, out_dev, cap, n_out_dev):
    return lib().dm_rebalance_async(h, _ptr(out_dev), cap, _ptr(n_out_dev))


def dm_commit_cache(h):
    return lib().dm_commit_cache(h)


def dm_hash_prompts(h, batch, keys_dev, key_off_dev, pos_dev):
    return lib().dm_hash_prompts(h, C.byref(batch), _ptr(keys_dev), _ptr(key_off_dev), _ptr(pos_dev))


def dm_hash_prompts_noalloc(block_tokens, route_prefix_blocks, seed, batch, keys_dev, key_off_dev, pos_dev,
                            stream=None):
    return lib().dm_hash_prompts_noalloc(block_tokens, route_prefix_blocks, seed, C.byref(batch), _ptr(keys_dev),
                                         _ptr(key_off_dev), _ptr(pos_dev), stream)


def dm_ring_lookup(h, pos_dev, n, owner1_dev, owner2_dev):
    return lib().dm_ring_lookup(h, _ptr(pos_dev), n, _ptr(owner1_dev), _ptr(owner2_dev))


def dm_get_loads(h, M):
    W = np.zeros(M, np.uint64)
    n = C.c_uint32()
    _check(lib().dm_get_loads(h, W.ctypes.data, M, C.byref(n)), "dm_get_loads")
    return W[:min(M, n.value)]


def dm_export_cache(h, i):
    n = C.c_uint64()
    _check(lib().dm_export_cache(h, i, None, None, 0, C.byref(n)), "dm_export_cache")
    k = np.zeros(max(n.value, 1), np.uint64)
    s = np.zeros(max(n.value, 1), np.uint64)
    _check(lib().dm_export_cache(h, i, k.ctypes.data, s.ctypes.data, n.value, C.byref(n)), "dm_export_cache")
    return k[:n.value], s[:n.value]


def dm_export_queue(h, i, cap=1 << 20):
    n = C.c_uint64()
    seq = np.zeros(cap, np.uint64)
    work = np.zeros(cap, np.uint64)
    rem = np.zeros(cap, np.uint64)
    _check(lib().dm_export_queue(h, i, seq.ctypes.data, work.ctypes.data, rem.ctypes.data, cap, C.byref(n)),
           "dm_export_queue")
    m = min(n.value, cap)
    return seq[:m], work[:m], rem[:m]


def dm_export_ring(h, f, cap):
    n = C.c_uint32()
    vp = np.zeros(max(cap, 1), np.uint64)
    ow = np.zeros(max(cap, 1), np.uint32)
    _check(lib().dm_export_ring(h, f, vp.ctypes.data, ow.ctypes.data, cap, C.byref(n)), "dm_export_ring")
    m = min(n.value, cap)
    return vp[:m], ow[:m]


def dm_get_clock(h):
    c = C.c_uint64()
    _check(lib().dm_get_clock(h, C.byref(c)), "dm_get_clock")
    return c.value


def dm_get_maint_counts(h):
    """(index rebuilds, log compactions) since the handle was created."""
    a, b = C.c_uint64(), C.c_uint64()
    _check(lib().dm_get_maint_counts(h, C.byref(a), C.byref(b)), "dm_get_maint_counts")
    return a.value, b.value


def dm_get_metrics(h, reset=False):
    """(dict of dm_metrics fields, TTFT histogram counts)."""
    m = dm_metrics()
    hist = np.zeros(DM_HIST_BUCKETS, np.uint64)
    _check(lib().dm_get_metrics(h, C.byref(m), hist.ctypes.data, DM_HIST_BUCKETS, 1 if reset else 0),
           "dm_get_metrics")
    return {name: getattr(m, name) for name, _ in dm_metrics._fields_}, hist


def dm_get_route_blocks(h, out_dev, n):
    return lib().dm_get_route_blocks(h, _ptr(out_dev), n)


def dm_export_prefix_tree(h):
    """Keys of the expanded nodes of the adaptive prefix tree (sorted)."""
    n = C.c_uint64()
    _check(lib().dm_export_prefix_tree(h, None, 0, C.byref(n)), "dm_export_prefix_tree")
    k = np.zeros(max(n.value, 1), np.uint64)
    _check(lib().dm_export_prefix_tree(h, k.ctypes.data, n.value, C.byref(n)), "dm_export_prefix_tree")
    return np.sort(k[:n.value])


def dm_potc_max_loads(n_bins, m_balls, d, trials, seed, max_load_dev, stream=None):
    return lib().dm_potc_max_loads(n_bins, m_balls, d, trials, seed, _ptr(max_load_dev), stream)


def dm_last_error(h):
    return lib().dm_last_error(h)


DM_PROFILE_ONLY = 0x100


def dm_set_profiling(h, on, stages=None):
    """on: time every stage; stages: names of STAGES to time instead (others untimed)."""
    if stages is not None:
        mode = DM_PROFILE_ONLY
        for name in stages:
            mode |= 1 << STAGES.index(name)
        return lib().dm_set_profiling(h, mode)
    return lib().dm_set_profiling(h, 1 if on else 0)


def dm_get_stage_times(h, reset=False):
    ms = np.zeros(len(STAGES), np.float64)
    calls = np.zeros(len(STAGES), np.uint64)
    _check(lib().dm_get_stage_times(h, ms.ctypes.data, calls.ctypes.data, 1 if reset else 0),
           "dm_get_stage_times")
    return {s: (float(ms[i]), int(calls[i])) for i, s in enumerate(STAGES)}
