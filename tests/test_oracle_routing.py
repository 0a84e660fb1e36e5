"""Pins of the oracle's routing state machine: the ring example of App. A.1.3,
brute-force ring scans, add/remove locality, the distinct-candidate equation,
hand-built cases of the SLO rule, queue draining, exact LRU against a top-C
recomputation, prefix closure, the cache-affinity guarantee of Sec. 2.3, the
power-of-two-choices effect, hand-built rebalancing, and argument errors."""

import json
import os

import numpy as np
import pytest

from oracle import oracle as O
from tracegen import Trace, workload

GOLD = os.path.join(os.path.dirname(__file__), "golden")


def mk(M=8, V=16, C=1 << 16, slo=10**6, B=16, K=16, seed=3, live=None, max_batch=4096):
    o = O.Oracle(block_tokens=B, route_prefix_blocks=K, vnodes_per_instance=V, max_instances=M,
                 cache_capacity_blocks=C, slo_us=slo, cost_us_per_token=1, hot_num=3, hot_den=2,
                 max_batch=max_batch, max_batch_tokens=1 << 30, seed=seed)
    for i in (range(M) if live is None else live):
        assert o.add_instance(i) == 0
    return o


def brute_successor(vpos, p):
    idx = [i for i, x in enumerate(vpos) if x >= p]
    return min(idx, key=lambda i: (vpos[i], i)) if idx else 0


# -- rings --------------------------------------------------------------------

def test_ring_example_app_a13():
    g = json.load(open(os.path.join(GOLD, "ring_example.json")))
    for phase in ("before", "after"):
        pos = np.array(g[phase]["pos"], np.uint64)
        own = g[phase]["owner"]
        for pr in g["probes"]:
            assert own[O.ring_successor(pos, pr["p"])] == pr[phase], (phase, pr)


def test_ring_successor_vs_linear_scan():
    rng = np.random.default_rng(1)
    for R in (1, 2, 7, 64, 513):
        vpos = np.sort(rng.integers(0, 1000, size=R).astype(np.uint64))   # many ties
        for p in list(range(0, 1002, 7)) + [int(x) for x in vpos]:
            assert O.ring_successor(vpos, p) == brute_successor(vpos.tolist(), p)


def test_state_ring_layout():
    o = mk(M=6, V=9, live=[0, 2, 3, 5])
    _, _, sc = o.key_material()
    for f in (0, 1):
        vp, ow, vi = o.ring(f)
        assert len(vp) == 4 * 9
        recs = list(zip(vp.tolist(), ow.tolist(), vi.tolist()))
        assert recs == sorted(recs)
        assert set(ow.tolist()) == {0, 2, 3, 5}
        for p, i, v in recs:
            assert p == O.fmix64(O.mix64((i << 32) | v) ^ int(sc[5 + f]))


def test_ring_owners_vs_brute_force():
    o = mk(M=8, V=5)
    rng = np.random.default_rng(2)
    pos = rng.integers(0, 2**63, size=300, dtype=np.int64).astype(np.uint64) * np.uint64(2)
    for f in (0, 1):
        vp, ow, _ = o.ring(f)
        got = o.ring_owners(pos, f)
        want = [int(ow[brute_successor(vp.tolist(), int(p))]) for p in pos]
        assert got.tolist() == want
        # a position equal to a vnode position belongs to that vnode
        assert o.ring_owners(vp, f).tolist() == ow.tolist()


def test_add_remove_locality():
    o = mk(M=12, V=8, live=range(10))
    rng = np.random.default_rng(5)
    pos = rng.integers(0, 2**63, size=4000, dtype=np.int64).astype(np.uint64) * np.uint64(2)
    before = [o.ring_owners(pos, f) for f in (0, 1)]
    assert o.add_instance(10) == 0
    after = [o.ring_owners(pos, f) for f in (0, 1)]
    for f in (0, 1):
        moved = before[f] != after[f]
        assert moved.any()
        assert np.all(after[f][moved] == 10)
    assert o.remove_instance(3) == 0
    after2 = [o.ring_owners(pos, f) for f in (0, 1)]
    for f in (0, 1):
        moved = after[f] != after2[f]
        assert moved.any()
        assert np.all(after[f][moved] == 3)
        assert not np.any(after2[f] == 3)


# -- distinct candidates ------------------------------------------------------

def test_next_live_dense_is_paper_formula():
    o = mk(M=8)
    for i in range(8):
        assert o.next_live(i) == (i + 1) % 8


def test_next_live_with_holes():
    o = mk(M=10, live=[1, 4, 5, 9])
    assert [o.next_live(i) for i in (1, 4, 5, 9)] == [4, 5, 9, 1]


def _route_trace(o, tr, b):
    s, e, off, lens, _ = tr.batch_layout(b)
    return o.route_batch(tr.batch_tokens(b), off, lens, tr.batch_time(b))


def test_candidates_distinct_and_raw():
    w = workload("tiny", n_requests=300, batch=300)
    tr = Trace(w)
    o = mk(M=8, V=64, seed=w["seed"])
    rc, out = _route_trace(o, tr, 0)
    assert rc == 0
    assert np.all(out["cand1"] != out["cand2"])
    pos = np.array([o.prompt_keys(tr.request_tokens(r))[1] for r in range(tr.n)])
    raw1, raw2 = o.ring_owners(pos[:, 0].copy(), 0), o.ring_owners(pos[:, 1].copy(), 1)
    assert np.array_equal(out["cand1"], raw1)
    coll = raw1 == raw2
    assert np.array_equal(out["cand2"][~coll], raw2[~coll])
    assert np.array_equal(out["cand2"][coll], (raw1[coll] + 1) % 8)


# -- the SLO-aware choice (Sec. 3.2) ------------------------------------------

@pytest.mark.parametrize("case", [
    # (c1,c2,h1,h2,L,W1,W2,slo) -> (chosen, switched)
    ((3, 5, 64, 64, 100, 10, 20, 10**6), (3, 0)),   # equal hits: less loaded
    ((3, 5, 64, 64, 100, 20, 10, 10**6), (5, 0)),
    ((3, 5, 64, 64, 100, 10, 10, 10**6), (3, 0)),   # equal hits, tie -> c1
    ((3, 5, 0, 0, 100, 7, 6, 0), (5, 0)),           # equal (zero) hits ignore the SLO
    ((3, 5, 80, 16, 100, 500, 0, 10**6), (3, 0)),   # affinity although c1 far more loaded
    ((3, 5, 16, 80, 100, 0, 500, 10**6), (5, 0)),   # mirrored
    ((3, 5, 80, 16, 100, 980, 0, 1000), (3, 0)),    # ttft_a == SLO exactly: keep affinity
    ((3, 5, 80, 16, 100, 981, 0, 1000), (5, 1)),    # ttft_a > SLO: less-loaded b
    ((3, 5, 80, 16, 100, 981, 981, 1000), (3, 1)),  # switched, tie -> a
    ((3, 5, 80, 16, 100, 981, 2000, 1000), (3, 1)), # switched but a is less loaded
    ((3, 5, 16, 80, 100, 0, 981, 1000), (3, 1)),    # mirrored switch to c1
])
def test_choice_rule_cases(case):
    (c1, c2, h1, h2, L, W1, W2, slo), want = case
    ch, t1, t2, sw = O.choose(c1, c2, h1, h2, L, W1, W2, slo)
    assert (ch, sw) == want
    assert t1 == W1 + (L - h1) and t2 == W2 + (L - h2)


def test_choice_differs_from_min_ttft():
    """App. A.1.1: Min-TTFT would move a request whose affine instance is
    slower but within the SLO; the SLO-aware rule keeps it."""
    ch, t1, t2, sw = O.choose(0, 1, 96, 0, 100, 400, 0, 10**6)
    assert t2 < t1 <= 10**6
    assert ch == 0 and sw == 0


def test_cost_scales_uncached_tokens():
    ch, t1, t2, sw = O.choose(0, 1, 32, 0, 100, 5, 9, 10**6, cost=3)
    assert t1 == 5 + 3 * 68 and t2 == 9 + 3 * 100


# -- queues and draining --------------------------------------------------------

def test_drain_fifo():
    o = mk(M=4)
    for s, w in enumerate([5, 3, 7]):
        o.debug_enqueue(0, s, 100, 0, 1, 0, 0, w)
    assert o.route_batch([], [], [], 1000)[0] == 0        # first batch: no drain
    assert o.queue(0)[2].tolist() == [5, 3, 7]
    assert o.route_batch([], [], [], 1006)[0] == 0        # 6 us: 5 done, 1 of 3
    seq, work, rem = o.queue(0)
    assert seq.tolist() == [1, 2] and rem.tolist() == [2, 7] and work.tolist() == [3, 7]
    assert int(o.loads()[0]) == 9
    assert o.route_batch([], [], [], 1100)[0] == 0
    assert len(o.queue(0)[0]) == 0 and int(o.loads()[0]) == 0


def test_drain_pops_zero_work_at_head():
    o = mk(M=4)
    o.debug_enqueue(1, 0, 16, 0, 1, 16, 0, 0)
    o.debug_enqueue(1, 1, 16, 0, 1, 0, 0, 4)
    o.route_batch([], [], [], 0)
    o.route_batch([], [], [], 0)
    assert o.queue(1)[0].tolist() == [1]


# -- commit: exact LRU ----------------------------------------------------------

def _run(o, tr, commit=True, rebalance=False):
    outs = []
    for b in range(len(tr.batches)):
        rc, out = _route_trace(o, tr, b)
        assert rc == 0
        if rebalance:
            assert o.rebalance()[0] == 0
        if commit:
            assert o.commit() == 0
        outs.append(out)
    return outs


def test_lru_equals_top_c_last_touch():
    """Sequential LRU of capacity C == the C distinct keys with the latest
    last touch (recomputed from the trace, touches in the commit order)."""
    w = workload("tiny", n_requests=400, batch=50)
    tr = Trace(w)
    C = 300
    o = mk(M=8, V=64, C=C, seed=w["seed"])
    outs = _run(o, tr)
    chosen = np.concatenate([x["chosen"] for x in outs])
    last = {}
    stamp = 0
    for r in range(tr.n):
        keys, _ = o.prompt_keys(tr.request_tokens(r))
        for b in range(len(keys) - 1, -1, -1):
            stamp += 1
            last[(int(chosen[r]), int(keys[b]))] = stamp
    assert o.clock() == stamp
    for i in range(8):
        mine = sorted(((s, k) for (j, k), s in last.items() if j == i), reverse=True)[:C]
        k, s = o.cache(i)
        assert sorted(zip(s.tolist(), k.tolist()), reverse=True) == mine


def test_prefix_closed_and_hits_are_leading_runs():
    """Descending touch order keeps every resident set prefix-closed, so the
    leading run equals the longest resident prefix found by any search."""
    w = workload("tiny", n_requests=512, batch=64)
    tr = Trace(w)
    o = mk(M=8, V=64, C=500, seed=w["seed"])
    _run(o, tr)
    res = [set(o.cache(i)[0].tolist()) for i in range(8)]
    for r in range(0, tr.n, 3):
        keys, _ = o.prompt_keys(tr.request_tokens(r))
        for i in range(8):
            flags = [int(k) in res[i] for k in keys]
            run = flags.index(False) if False in flags else len(flags)
            assert not any(flags[run:]), (r, i)


def test_capacity_below_one_request():
    """C smaller than a prompt's block count keeps blocks 0..C-1 (touched last)."""
    o = mk(M=2, C=5)
    tok = np.arange(16 * 12, dtype=np.uint32)
    assert o.route_batch(tok, [0], [len(tok)], 0)[0] == 0
    assert o.commit() == 0
    rc, out = o.route_batch(tok, [0], [len(tok)], 0)
    assert rc == 0
    assert sorted([int(out["hit1"][0]), int(out["hit2"][0])]) == [0, 5 * 16]


def test_probe_sees_batch_start_state():
    """Two identical prompts in one batch: neither sees the other's blocks."""
    o = mk(M=4)
    tok = np.arange(16 * 8, dtype=np.uint32)
    rc, out = o.route_batch(np.concatenate([tok, tok]), [0, 128], [128, 128], 0)
    assert rc == 0 and out["hit1"].tolist() == [0, 0] and out["hit2"].tolist() == [0, 0]
    o.commit()
    rc, out = o.route_batch(tok, [0], [128], 0)
    assert max(out["hit1"][0], out["hit2"][0]) == 128


def test_cache_affinity_guarantee_sec23():
    """Batch size 1, no eviction, no SLO pressure: a group of m requests with
    one prefix sees at most 2 cold misses (Sec. 2.3: hit rate >= 1 - 2/m)."""
    o = mk(M=8, C=1 << 20, slo=1 << 60)
    rng = np.random.default_rng(8)
    prefixes = [rng.integers(0, 32000, size=16 * 20, dtype=np.uint32) for _ in range(6)]
    misses = [0] * 6
    t = 0
    for r in range(120):
        g = r % 6
        tok = np.concatenate([prefixes[g], rng.integers(0, 32000, size=40, dtype=np.uint32)])
        rc, out = o.route_batch(tok, [0], [len(tok)], t)
        assert rc == 0
        h = out["hit1"][0] if out["chosen"][0] == out["cand1"][0] else out["hit2"][0]
        misses[g] += int(h < 16 * 20)
        o.commit()
        t += 1
    assert max(misses) <= 2


def test_two_choices_flatten_load():
    """Power of two choices (Sec. 2.3): with no cache reuse, picking the less
    loaded of two ring candidates keeps the max load far closer to the mean
    than the first candidate alone."""
    w = workload("tiny", n_requests=4000, batch=500, n_prefix=4000, prefix_lo=2048, prefix_hi=2048,
                 len_lo=256, len_hi=256)
    tr = Trace(w)
    o = mk(M=16, V=64, C=1, slo=1 << 60, seed=w["seed"])
    outs = []
    for b in range(len(tr.batches)):
        s, e, off, lens, _ = tr.batch_layout(b)
        rc, out = o.route_batch(tr.batch_tokens(b), off, lens, 0)
        assert rc == 0
        outs.append(out)
    W = o.loads()[:16].astype(np.float64)
    single = np.bincount(np.concatenate([x["cand1"] for x in outs]), minlength=16) * 256.0
    dev2 = W.max() - W.mean()
    dev1 = single.max() - single.mean()
    assert dev2 < 0.25 * dev1


# -- rebalancing (Sec. 3.3) -----------------------------------------------------

def test_rebalance_hand_built():
    """Instance 0 holds 1,000 us of queued work, 1..3 hold 0; 2*4*W_0 > 3*sum.
    Queue of 0 (head first), L=100 each:
      seq 10: work 100 (c1=0,c2=1,h1=0,h2=0)  B = 100 - 100        = 0   -> no
      seq 11: work 300 (c1=0,c2=2,h1=0,h2=90) B = 400 - 10         = 390
      seq 12: work 200 (c1=3,c2=0,h1=50,h2=0) B = 600 - 50         = 550
      seq 13: work 400 (c1=0,c2=1,h1=0,h2=0)  B = 1000 - 100       = 900
    Order by B desc: 13, 12, 11.  Migrate 13 -> 1 (W0=600, W1=100);
    0 still hot (8*600 > 3*1000); migrate 12 -> 3 (W0=400, W3=50,
    sum=550; 8*400 > 3*550); migrate 11 -> 2 (W0=100, W2=10, sum=260;
    8*100 > 3*260 = 780: still hot, but no candidates left)."""
    o = mk(M=4, slo=10**6)
    o.debug_enqueue(0, 10, 100, 0, 1, 0, 0, 100)
    o.debug_enqueue(0, 11, 100, 0, 2, 0, 90, 300)
    o.debug_enqueue(0, 12, 100, 3, 0, 50, 0, 200)
    o.debug_enqueue(0, 13, 100, 0, 1, 0, 0, 400)
    rc, n, (seq, fr, to) = o.rebalance()
    assert rc == 0 and n == 3
    assert seq.tolist() == [13, 12, 11] and fr.tolist() == [0, 0, 0] and to.tolist() == [1, 3, 2]
    assert o.loads()[:4].tolist() == [100, 100, 10, 50]
    assert o.queue(0)[0].tolist() == [10]
    assert o.queue(1)[1].tolist() == [100] and o.queue(3)[1].tolist() == [50]


def test_rebalance_respects_slo_and_stop():
    """A target whose TTFT would reach the SLO is skipped; migration stops as
    soon as the source is no longer a hotspot."""
    o = mk(M=4, slo=150)
    o.debug_enqueue(0, 1, 100, 0, 1, 0, 0, 300)   # B = 300-100 = 200, ttft_j = 100 < 150 -> move
    o.debug_enqueue(0, 2, 100, 0, 2, 0, 0, 300)   # would move, but 0 is no longer hot? check
    o.debug_enqueue(0, 3, 200, 0, 3, 0, 0, 300)   # ttft_j = 200 >= SLO -> never
    # W0 = 900, sum 900: hot.  Order: seq 3 (B=900-200=700), seq 2 (600-100=500), seq 1 (200).
    rc, n, (seq, fr, to) = o.rebalance()
    # seq 3 skipped (SLO); seq 2 -> 2: W0=600, W2=100, sum=700, 8*600 > 2100 hot;
    # seq 1 -> 1: W0=300, W1=100, sum=500, 8*300=2400 > 1500 still hot; list exhausted.
    assert rc == 0 and seq.tolist() == [2, 1] and to.tolist() == [2, 1]
    o2 = mk(M=4, slo=10**6)
    o2.debug_enqueue(0, 1, 100, 0, 1, 0, 0, 50)
    o2.debug_enqueue(1, 2, 100, 1, 2, 0, 0, 50)
    o2.debug_enqueue(2, 3, 100, 2, 3, 0, 0, 50)
    o2.debug_enqueue(3, 4, 100, 3, 0, 0, 0, 50)
    assert o2.rebalance()[1] == 0                   # balanced: no hotspot


def test_rebalance_skips_started_and_conserves_work():
    # many Zipf prefixes + small batches: affinity piles one prefix group on
    # an instance whose other groups then have cool alternatives
    w = workload("scaling", n_requests=3000, batch=50, n_instances=16, vnodes=32, n_prefix=100,
                 zipf_s=1.2, len_lo=400, len_hi=512, prefix_lo=384, prefix_hi=384, scale_every=0,
                 rho=1.0)
    tr = Trace(w)
    o = mk(M=16, V=32, C=4096, slo=10**9, seed=w["seed"])
    total_moves = 0
    for b in range(len(tr.batches)):
        rc, out = _route_trace(o, tr, b)
        assert rc == 0
        before = {i: o.queue(i) for i in range(16)}
        rc, n, (seq, fr, to) = o.rebalance()
        assert rc == 0
        total_moves += n
        for s_, f_, t_ in zip(seq.tolist(), fr.tolist(), to.tolist()):
            bs, bw, br = before[f_]
            k = bs.tolist().index(s_)
            assert bw[k] == br[k]                    # only not-started requests move
            assert s_ in o.queue(t_)[0].tolist()
        W = o.loads()
        for i in range(16):
            assert int(W[i]) == int(o.queue(i)[2].sum())
        o.commit()
    assert total_moves > 0


# -- errors -----------------------------------------------------------------------

def test_errors():
    o = mk(M=4, live=[0])
    assert o.route_batch(np.zeros(16, np.uint32), [0], [16], 0)[0] == O.ERR_NO_INSTANCES
    assert o.add_instance(0) == O.ERR_DUPLICATE_ID
    assert o.add_instance(7) == O.ERR_INVALID_ARG
    assert o.remove_instance(2) == O.ERR_UNKNOWN_ID
    assert o.add_instance(1) == 0
    assert o.route_batch(np.zeros(16, np.uint32), [0], [15], 0)[0] == O.ERR_INVALID_ARG
    assert o.route_batch(np.zeros(32, np.uint32), [0], [16], 10)[0] == 0
    assert o.route_batch(np.zeros(32, np.uint32), [0], [16], 9)[0] == O.ERR_ORDER
    # a removed instance with queued work cannot be re-added until drained
    _, out = o.route_batch(np.zeros(32, np.uint32), [0], [32], 10)
    busy = int(out["chosen"][0])
    assert o.remove_instance(busy) == 0
    assert o.add_instance(busy) == O.ERR_DUPLICATE_ID
    o.add_instance(2)
    o.route_batch([], [], [], 10**6)
    assert o.add_instance(busy) == 0
    o5 = mk(M=4, max_batch=2)
    assert o5.route_batch(np.zeros(48, np.uint32), [0, 16, 32], [16, 16, 16], 0)[0] == O.ERR_CAPACITY
