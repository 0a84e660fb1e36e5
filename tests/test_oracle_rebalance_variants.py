"""Pins of the oracle's rebalancing variants, the paper's own wording of
hotspot-aware rebalancing (Sec. 3.3, App. A.1.2): migrate "until all
requests in the overloaded instance's queue are expected to meet the TTFT
SLO" (overloaded = queued work above the SLO), and start migrating "whenever
both candidate instances of a request are identified as overloaded".
Expected values are worked out by hand."""

import numpy as np

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
