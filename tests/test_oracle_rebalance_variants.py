"""Pins of the oracle's rebalancing variants, the paper's own wording of
hotspot-aware rebalancing (Sec. 3.3, App. A.1.2): migrate "until all
requests in the overloaded instance's queue are expected to meet the TTFT
SLO" (overloaded = queued work above the SLO), start migrating "whenever
both candidate instances of a request are identified as overloaded", and
estimate a candidate's TTFT on the other instance from that instance's
cache as it stands at the call (fresh hits) rather than from the hit
stored at routing time.  Expected values are worked out by hand."""

import numpy as np
import pytest

from oracle import oracle as O


def mk(flags, slo, M=4):
    o = O.Oracle(block_tokens=16, route_prefix_blocks=4, vnodes_per_instance=16, max_instances=M,
                 cache_capacity_blocks=1 << 12, slo_us=slo, cost_us_per_token=1, hot_num=3, hot_den=2,
                 max_batch=16, max_batch_tokens=1 << 16, seed=5, rebalance_flags=flags)
    for i in range(M):
        assert o.add_instance(i) == 0
    return o


def four_entries(o):
    """Instance 0: four entries of 100 us (L = 100, no hits), alternatives
    1, 3, 2, 1... in queue order: seq 1 -> j 1, 2 -> 2, 3 -> 3, 4 -> 1."""
    for seq, j in ((1, 1), (2, 2), (3, 3), (4, 1)):
        o.debug_enqueue(0, seq, 100, 0, j, 0, 0, 100)


def test_slo_target_stops_once_the_queue_meets_the_slo():
    """W0 = 400, SLO 250.  Benefits (TTFT on 0 minus 0 + 100 on j): seq 4
    300, seq 3 200, seq 2 100, seq 1 0.  SLO target: move 4 (W0 300 > 250),
    move 3 (W0 200), then W0 <= 250: stop.  Default rule (hot while
    2*4*W0 > 3*sum): 4, 3 and 2 move (8*200 = 1600 > 1200), then
    8*100 = 800 <= 1200 stops."""
    o = mk(O.RB_SLO_TARGET, 250)
    four_entries(o)
    rc, n, (seq, fr, to) = o.rebalance()
    assert rc == 0 and seq.tolist() == [4, 3] and to.tolist() == [1, 3]
    assert o.loads().tolist() == [200, 100, 0, 100]
    o = mk(0, 250)
    four_entries(o)
    rc, n, (seq, fr, to) = o.rebalance()
    assert rc == 0 and seq.tolist() == [4, 3, 2] and to.tolist() == [1, 3, 2]


def test_slo_target_ignores_hot_instances_within_the_slo():
    """W0 = 200 (others 0) is a hotspot by the 1.5x-mean rule but meets a
    250 us SLO: the SLO target moves nothing, the default rule moves."""
    for flags, want in ((O.RB_SLO_TARGET, 0), (0, 1)):
        o = mk(flags, 250)
        o.debug_enqueue(0, 1, 100, 0, 1, 0, 0, 100)
        o.debug_enqueue(0, 2, 100, 0, 2, 0, 0, 100)
        assert o.rebalance()[1] == want


def _prompt_with_candidates(o, want, seed=3):
    rng = np.random.default_rng(seed)
    for _ in range(2000):
        t = rng.integers(0, 32000, 64, dtype=np.uint32)
        _, pos = o.prompt_keys(t)
        c1 = int(o.ring_owners(pos[:1], 0)[0])
        raw2 = int(o.ring_owners(pos[1:], 1)[0])
        c2 = raw2 if raw2 != c1 else int(o.next_live(c1))
        if {c1, c2} == want:
            return t
    raise AssertionError("no prompt found")


def _loaded(flags):
    """W0 = 3,000 (alternatives 2 and 3, idle), W1 = 1,000; SLO 500."""
    o = mk(flags, 500)
    assert o.route_batch([], [], [], 0)[0] == 0
    o.debug_enqueue(0, 100, 100, 0, 2, 0, 0, 1000)
    o.debug_enqueue(0, 101, 100, 3, 0, 0, 0, 2000)
    o.debug_enqueue(1, 102, 100, 1, 2, 0, 0, 1000)
    return o


def test_double_overload_trigger_gates_the_rule():
    """After a batch whose request has candidates {2, 3} (idle: TTFT 64 <=
    500) the triggered variant moves nothing; after one whose request has
    candidates {0, 1} (TTFT >= 1,000 on both) it moves exactly what the
    untriggered rule moves on the same state."""
    probe = _loaded(0)
    quiet = _prompt_with_candidates(probe, {2, 3})
    loud = _prompt_with_candidates(probe, {0, 1})
    results = {}
    for name, prompt in (("quiet", quiet), ("loud", loud)):
        for flags in (0, O.RB_DOUBLE_OVERLOAD):
            o = _loaded(flags)
            rc, out = o.route_batch(prompt, [0], [64], 0)
            assert rc == 0
            both = out["ttft1"][0] > 500 and out["ttft2"][0] > 500
            assert both == (name == "loud")
            rc, n, (seq, fr, to) = o.rebalance()
            assert rc == 0
            results[name, flags] = (seq.tolist(), to.tolist())
    assert results["quiet", O.RB_DOUBLE_OVERLOAD] == ([], [])
    assert results["quiet", 0][0]                       # the untriggered rule moves
    assert results["loud", O.RB_DOUBLE_OVERLOAD] == results["loud", 0]
    assert results["loud", 0][0]


def test_fresh_hits_see_a_prefix_cached_after_routing():
    """Request X (4 blocks, 64 tokens) is routed while nothing is cached: both
    stored hits are 0 and it queues on i (equal hits: the less loaded, tie
    c1).  Behind it on i an entry B of 1,000 us (alternative 2, no hits).
    After the commit, X's four keys are also touched on its other candidate
    j.  Stored hits: X's benefit on j is 64 - (0 + 64) = 0 and B's 1,064 -
    1,000 = 64, so only B moves (then W_i = 64 is still hot, and X's move
    would not lower its TTFT).  Fresh hits: X's hit on j is 64 tokens, so
    its TTFT there is 0 and its benefit 64, tied with B's and first by
    sequence number: X moves to j, then B moves to 2."""
    probe = mk(0, 10 ** 9)
    prompt = _prompt_with_candidates(probe, {0, 1})
    keys, _ = probe.prompt_keys(prompt)
    results = {}
    for flags in (0, O.RB_FRESH_HITS):
        o = mk(flags, 10 ** 9)
        rc, out = o.route_batch(prompt, [0], [64], 0)
        assert rc == 0 and int(out["hit1"][0]) == int(out["hit2"][0]) == 0
        i = int(out["chosen"][0])
        j = int(out["cand2"][0]) if i == int(out["cand1"][0]) else int(out["cand1"][0])
        assert i == int(out["cand1"][0])
        assert o.commit() == 0
        for k in keys:
            assert o.debug_touch(j, int(k)) == 0
        o.debug_enqueue(i, 100, 1000, i, 2, 0, 0, 1000)
        rc, n, (seq, fr, to) = o.rebalance()
        assert rc == 0
        results[flags] = list(zip(seq.tolist(), fr.tolist(), to.tolist())), o.loads().tolist()
        xseq = 0
        if flags:
            assert results[flags][0] == [(xseq, i, j), (100, i, 2)]
            assert results[flags][1][j] == 0 and results[flags][1][2] == 1000 and results[flags][1][i] == 0
        else:
            assert results[flags][0] == [(100, i, 2)]
            assert results[flags][1][i] == 64 and results[flags][1][2] == 1000


def test_fresh_hits_equal_stored_hits_before_any_commit():
    """Between a batch's routing and its commit the caches do not change, so
    the fresh and the stored hits agree and so do the migrations."""
    from tracegen import Trace, workload
    w = workload("tiny", n_requests=400, batch=100, capacity=2000, zipf_s=1.3, rho=1.5)
    tr = Trace(w)
    got = {}
    for flags in (0, O.RB_FRESH_HITS):
        o = O.Oracle(**O.config_from_workload(w), rebalance_flags=flags)
        for i in range(w["n_instances"]):
            assert o.add_instance(i) == 0
        s, e, off, lens, nt = tr.batch_layout(0)
        assert o.route_batch(tr.batch_tokens(0), off, lens, tr.batch_time(0))[0] == 0
        rc, n, (seq, fr, to) = o.rebalance()
        assert rc == 0
        got[flags] = (seq.tolist(), to.tolist(), o.loads().tolist())
    assert got[0] == got[O.RB_FRESH_HITS]


def _model_rebalance(queues, live, flags, both_over, slo, cost, call, cached=None, B=16, seen=None):
    """Hotspot-aware rebalancing written out again in plain Python.  With
    RB_FRESH_HITS a candidate's hit on j is B x the leading run of its keys
    in cached[j] (instance j's resident keys at the call)."""
    W = {i: sum(e["rem"] for e in q) for i, q in queues.items()}
    if flags & O.RB_DOUBLE_OVERLOAD and not both_over:
        return []
    N = len(live)
    sumW = sum(W[i] for i in live)

    def over(i):
        return W[i] > slo if flags & O.RB_SLO_TARGET else 2 * N * W[i] > 3 * sumW

    def hit_of(e, j):
        stored = e["h1"] if j == e["c1"] else e["h2"]
        if not flags & O.RB_FRESH_HITS:
            return stored
        run = 0
        while run < len(e["keys"]) and int(e["keys"][run]) in cached[j]:
            run += 1
        if seen is not None and B * run != stored:
            seen.append(e["seq"])
        return B * run

    hot = sorted((i for i in live if over(i)), key=lambda i: (-W[i], i))
    moves = []
    for i in hot:
        ahead, cands = 0, []
        for e in queues[i]:
            ttft_i = ahead + e["rem"]
            ahead += e["rem"]
            if e["rem"] != e["work"] or e["moved"] == call:
                continue
            j = e["c2"] if e["c1"] == i else e["c1"]
            hj = hit_of(e, j)
            cands.append((-(ttft_i - (W[j] + cost * (e["L"] - hj))), e["seq"], ttft_i))
        for _, seq, ttft_i in sorted(cands):
            if not over(i):
                break
            e = next(x for x in queues[i] if x["seq"] == seq)
            j = e["c2"] if e["c1"] == i else e["c1"]
            if j not in live:
                continue
            hj = hit_of(e, j)
            nw = cost * (e["L"] - hj)
            if not (ttft_i > W[j] + nw and W[j] + nw < slo):
                continue
            queues[i].remove(e)
            W[i] -= e["work"]
            sumW -= e["work"]
            e.update(work=nw, rem=nw, moved=call)
            queues[j].append(e)
            W[j] += nw
            sumW += nw
            moves.append((seq, i, j))
    return moves


@pytest.mark.parametrize("flags", [0, O.RB_SLO_TARGET, O.RB_DOUBLE_OVERLOAD, 3, O.RB_FRESH_HITS,
                                   O.RB_FRESH_HITS | O.RB_SLO_TARGET])
def test_variants_match_an_independent_model_on_a_trace(flags):
    """A skewed 16-instance workload with a 5 ms SLO, rebalancing after
    every batch: the migrations of every call and the loads after it equal
    an independent model of the queues and of the rule, and the completion
    TTFTs (migrated requests keep their arrival) equal the oracle's
    metrics."""
    from tracegen import Trace, workload
    w = workload("scaling", n_requests=3000, batch=50, n_instances=16, vnodes=32, n_prefix=100, zipf_s=1.2,
                 len_lo=400, len_hi=512, prefix_lo=384, prefix_hi=384, scale_every=0, rho=1.0, slo_us=5000)
    tr = Trace(w)
    n, cost, slo = 16, w["cost_us"], w["slo_us"]
    o = O.Oracle(**O.config_from_workload(w, max_instances=n), rebalance_flags=flags)
    for i in range(n):
        assert o.add_instance(i) == 0
    queues = {i: [] for i in range(n)}
    live = set(range(n))
    t_prev, seq, total, ttfts, seen = None, 0, 0, [], []
    for b in range(len(tr.batches)):
        s, e, off, lens, nt = tr.batch_layout(b)
        t = tr.batch_time(b)
        if t_prev is not None:
            for q in queues.values():
                left, run = t - t_prev, 0
                while q and q[0]["rem"] <= left - run:
                    x = q.pop(0)
                    run += x["rem"]
                    ttfts.append(t_prev + run - x["arr"])   # a migrated request keeps its arrival
                if q:
                    q[0]["rem"] -= left - run
        t_prev = t
        rc, out = o.route_batch(tr.batch_tokens(b), off, lens, t)
        assert rc == 0
        both = False
        for r in range(len(lens)):
            c1, c2, ch = int(out["cand1"][r]), int(out["cand2"][r]), int(out["chosen"][r])
            h1, h2, L = int(out["hit1"][r]), int(out["hit2"][r]), int(lens[r])
            wk = cost * (L - (h1 if ch == c1 else h2))
            keys = o.prompt_keys(tr.request_tokens(s + r))[0] if flags & O.RB_FRESH_HITS else []
            queues[ch].append(dict(seq=seq, L=L, c1=c1, c2=c2, h1=h1, h2=h2, work=wk, rem=wk, moved=0, arr=t,
                                   keys=keys))
            both |= int(out["ttft1"][r]) > slo and int(out["ttft2"][r]) > slo
            seq += 1
        cached = {i: set(o.cache(i)[0].tolist()) for i in range(n)} if flags & O.RB_FRESH_HITS else None
        want = _model_rebalance(queues, live, flags, both, slo, cost, b + 1, cached, w["block_tokens"], seen)
        rc, nm, (mseq, mfr, mto) = o.rebalance()
        assert rc == 0
        assert list(zip(mseq.tolist(), mfr.tolist(), mto.tolist())) == want, b
        assert o.loads()[:n].tolist() == [sum(x["rem"] for x in queues[i]) for i in range(n)], b
        total += len(want)
        assert o.commit() == 0
    assert total > 0
    if flags & O.RB_FRESH_HITS:
        assert seen          # some candidate's fresh hit differed from its stored one
    m, _ = o.metrics()
    assert (m["completed"], m["ttft_sum_us"], m["ttft_max_us"]) == (len(ttfts), sum(ttfts), max(ttfts))
    assert m["slo_met"] == sum(x <= slo for x in ttfts)
