"""Pins of the oracle's policy variants and simulator metrics: hand-built cases
of each compared choice rule (Sec. 2.2, the ablation of Sec. 4.3 and the
related-work appendix), the TTFT histogram against brute force, completion
TTFTs of a hand-built queue, the load CV of Sec. 2.2 against numpy, counter
identities, and the qualitative ordering of the rules that Sec. 2.2 reports
(cache affinity reuses more, least loaded balances better)."""

import numpy as np
import pytest

from oracle import oracle as O
from tracegen import Trace, workload

AFF, LL, MT, PRE, DM = (O.RULE_CACHE_AFFINITY, O.RULE_LEAST_LOADED, O.RULE_MIN_TTFT, O.RULE_PREBLE,
                        O.RULE_DUALMAP)
GAFF, GLL, GMT, GPRE = (O.RULE_GLOBAL_CACHE_AFFINITY, O.RULE_GLOBAL_LEAST_LOADED, O.RULE_GLOBAL_MIN_TTFT,
                        O.RULE_GLOBAL_PREBLE)
ALL_RULES = [DM, AFF, LL, MT, PRE, GAFF, GLL, GMT, GPRE]


# -- the compared choice rules -------------------------------------------------

@pytest.mark.parametrize("case", [
    # (rule, c1, c2, h1, h2, L, W1, W2, slo) -> (chosen, switched)
    ((AFF, 3, 5, 80, 16, 100, 10**9, 0, 1000), (3, 0)),   # more hits wins however loaded
    ((AFF, 3, 5, 16, 80, 100, 0, 10**9, 1000), (5, 0)),
    ((AFF, 3, 5, 64, 64, 100, 20, 10, 1000), (5, 0)),     # equal hits: less loaded
    ((AFF, 3, 5, 64, 64, 100, 10, 10, 1000), (3, 0)),     # equal hits and loads: c1
    ((LL, 3, 5, 80, 16, 100, 11, 10, 10**6), (5, 1)),     # hits ignored: fewer hits chosen
    ((LL, 3, 5, 16, 80, 100, 10, 10, 10**6), (3, 1)),     # tie -> c1 although c2 has more hits
    ((LL, 3, 5, 16, 80, 100, 10, 11, 10**6), (3, 1)),
    ((LL, 3, 5, 0, 0, 100, 10, 9, 10**6), (5, 0)),        # equal hits never count as switched
    ((MT, 3, 5, 80, 16, 100, 70, 0, 10**6), (5, 1)),      # ttft 90 vs 84
    ((MT, 3, 5, 80, 16, 100, 64, 0, 10**6), (3, 0)),      # ttft 84 vs 84: tie -> c1
    ((MT, 3, 5, 16, 80, 100, 0, 64, 10**6), (3, 1)),      # 84 vs 84: tie -> c1 with fewer hits
    ((MT, 3, 5, 16, 80, 100, 0, 63, 10**6), (5, 0)),      # 84 vs 83
    ((PRE, 3, 5, 64, 0, 100, 10**6, 0, 1000), (3, 0)),    # 64% hit > 50%: affinity
    ((PRE, 3, 5, 48, 0, 96, 10**6, 0, 1000), (5, 1)),     # exactly 50%: not above, min TTFT
    ((PRE, 3, 5, 48, 0, 100, 60, 0, 1000), (5, 1)),       # 48%: min TTFT, 112 vs 100
    ((PRE, 3, 5, 48, 0, 100, 40, 0, 1000), (3, 0)),       # 48%: min TTFT, 92 vs 100
    ((PRE, 3, 5, 64, 64, 100, 5, 4, 1000), (5, 0)),       # both above half, equal: less loaded
])
def test_compared_rules(case):
    (rule, c1, c2, h1, h2, L, W1, W2, slo), want = case
    ch, t1, t2, sw = O.choose(c1, c2, h1, h2, L, W1, W2, slo, rule=rule)
    assert (ch, sw) == want
    assert t1 == W1 + (L - h1) and t2 == W2 + (L - h2)


def test_dualmap_rule_is_default_and_unchanged():
    """The SLO-aware rule of Sec. 3.2 keeps its own switched meaning: the
    switch fired, even where the higher-hit candidate is also less loaded."""
    assert O.choose(3, 5, 80, 16, 100, 981, 2000, 1000) == (3, 1001, 2084, 1)
    assert O.choose(3, 5, 80, 16, 100, 981, 2000, 1000, rule=DM) == (3, 1001, 2084, 1)


def test_rules_diverge_on_one_request():
    """One request separates all five rules (the contrasts the paper draws
    between DualMap and Min TTFT, cache affinity and least loaded): c1 holds
    60 of 100 tokens at load 500, c2 holds none at load 0, SLO 1000."""
    args = (0, 1, 60, 0, 100, 500, 0, 1000)
    got = {r: O.choose(*args, rule=r)[0] for r in (DM, AFF, LL, MT, PRE)}
    # DualMap: ttft_a = 540 <= SLO -> keep c1.  Affinity: c1.  Least loaded: c2.
    # Min TTFT: 540 vs 100 -> c2.  Preble: 60% > 50% -> affinity -> c1.
    assert got == {DM: 0, AFF: 0, LL: 1, MT: 1, PRE: 0}
    # below half the prompt Preble follows min TTFT
    assert O.choose(0, 1, 48, 0, 100, 500, 0, 1000, rule=PRE)[0] == 1


def test_dualmap_with_unbounded_slo_is_cache_affinity():
    """With an SLO no TTFT can exceed, the SLO-aware rule never switches and
    reduces to cache affinity (Sec. 3.2)."""
    rng = np.random.default_rng(5)
    for _ in range(2000):
        L = int(rng.integers(16, 400))
        h1, h2 = (int(x) * 16 for x in rng.integers(0, L // 16 + 1, 2))
        W1, W2 = (int(x) for x in rng.integers(0, 50, 2))
        a = O.choose(2, 7, h1, h2, L, W1, W2, 2**64 - 1)
        b = O.choose(2, 7, h1, h2, L, W1, W2, 2**64 - 1, rule=AFF)
        assert a == b


def test_unknown_rule_is_rejected():
    cfg = dict(block_tokens=16, route_prefix_blocks=4, vnodes_per_instance=4, max_instances=4,
               cache_capacity_blocks=64, slo_us=100, cost_us_per_token=1, hot_num=3, hot_den=2,
               max_batch=8, max_batch_tokens=1 << 16, seed=1)
    O.Oracle(**cfg, choice_rule=GPRE)
    with pytest.raises(ValueError):
        O.Oracle(**cfg, choice_rule=GPRE + 1)


# -- the rules over all live instances -------------------------------------------

def _global_case(rule, W, touched, L=64, absent=()):
    """Four instances with queued work W; instance i holds the first
    touched[i] blocks of a 64-token prompt (B = 16); one request routed."""
    o = O.Oracle(block_tokens=16, route_prefix_blocks=4, vnodes_per_instance=8, max_instances=5,
                 cache_capacity_blocks=64, slo_us=10**6, cost_us_per_token=1, hot_num=3, hot_den=2,
                 max_batch=8, max_batch_tokens=1 << 16, seed=7, choice_rule=rule)
    for i in range(5):
        assert o.add_instance(i) == 0
    for i in absent:
        assert o.remove_instance(i) == 0
    tok = np.arange(1000, 1000 + L, dtype=np.uint32)
    keys, _ = o.prompt_keys(tok)
    for i, nb in enumerate(touched):
        for k in keys[:nb][::-1]:
            assert o.debug_touch(i, int(k)) == 0
    assert o.route_batch([], [], [], 0)[0] == 0
    for i, w in enumerate(W):
        if w:
            o.debug_enqueue(i, 100 + i, L, i, i, 0, 0, w)
    rc, out = o.route_batch(tok, [0], [L], 0)
    assert rc == 0
    return o, out


def test_global_least_loaded():
    o, out = _global_case(GLL, [10, 3, 40, 3, 9], [0, 0, 4, 0, 0])
    assert out["chosen"][0] == 1 and out["switched"][0] == 0        # tie 3/3 -> lower id
    W = o.loads()
    assert W[1] == 3 + 64                                            # no hits on instance 1


def test_global_min_ttft():
    # keys: 10+64, 0+64, 40+32, 5+64, 80+0 -> instance 1
    o, out = _global_case(GMT, [10, 0, 40, 5, 80], [0, 0, 2, 0, 4])
    assert out["chosen"][0] == 1
    # instance 2 at load 20 holds 32 tokens: 20+32 = 52 < 64
    o, out = _global_case(GMT, [10, 0, 20, 5, 80], [0, 0, 2, 0, 4])
    assert out["chosen"][0] == 2 and o.loads()[2] == 20 + 32
    # instance 4 at load 52 holds the whole prompt: 52 + 0 ties 20 + 32 -> lower id
    o, out = _global_case(GMT, [10, 0, 20, 5, 52], [0, 0, 2, 0, 4])
    assert out["chosen"][0] == 2


def test_global_preble():
    # instance 4 holds the whole prompt (100% > 50%) although loaded
    o, out = _global_case(GPRE, [10, 0, 40, 5, 10**5], [0, 0, 2, 0, 4])
    assert out["chosen"][0] == 4 and o.loads()[4] == 10**5
    # two instances hold 3 of 4 blocks (75%): the less loaded of them
    o, out = _global_case(GPRE, [10, 0, 40, 5, 30], [0, 0, 3, 0, 3])
    assert out["chosen"][0] == 4
    # the best holds exactly half: min TTFT over all (0+64 on 1 vs 20+32 on 2)
    o, out = _global_case(GPRE, [10, 0, 20, 5, 80], [0, 0, 2, 0, 0])
    assert out["chosen"][0] == 2
    o, out = _global_case(GPRE, [10, 0, 40, 5, 80], [0, 0, 2, 0, 0])
    assert out["chosen"][0] == 1


def test_global_rules_skip_removed_instances():
    o, out = _global_case(GLL, [10, 3, 40, 3, 9], [0, 0, 4, 0, 0], absent=(1,))
    assert out["chosen"][0] == 3
    o, out = _global_case(GPRE, [10, 0, 40, 5, 10**5], [0, 0, 2, 0, 4], absent=(4,))
    assert out["chosen"][0] != 4


def test_global_cache_affinity_is_ring_one():
    for W in ([0, 0, 0, 0, 0], [10**6, 10**6, 10**6, 10**6, 10**6], [5, 0, 9, 1, 3]):
        o, out = _global_case(GAFF, W, [0, 4, 0, 2, 0])
        assert out["chosen"][0] == out["cand1"][0] and out["switched"][0] == 0


# -- TTFT histogram --------------------------------------------------------------

def test_histogram_buckets_brute_force():
    """Each value lies in [lower(k), lower(k+1)); values below 16 are exact;
    each bucket above is 1/16 of its power of two wide (relative width <=
    1/16)."""
    lows = [O.hist_lower(k) for k in range(O.HIST_BUCKETS)]
    assert lows[:17] == list(range(17))
    assert all(a < b for a, b in zip(lows, lows[1:]))
    assert lows[-1] == 31 << 59
    for k in range(16, O.HIST_BUCKETS - 1):
        assert (lows[k + 1] - lows[k]) * 16 <= lows[k]
    rng = np.random.default_rng(1)
    vals = [0, 1, 15, 16, 17, 31, 32, 33, 47, 48, 2**63, 2**64 - 1]
    vals += [int(x) for x in rng.integers(0, 2**63, 300, dtype=np.uint64)]
    vals += [int(x) >> int(s) for x, s in zip(rng.integers(0, 2**63, 300, dtype=np.uint64),
                                              rng.integers(0, 63, 300))]
    for v in vals:
        k = O.hist_bucket(v)
        assert lows[k] <= v
        assert k == O.HIST_BUCKETS - 1 or v < lows[k + 1]


# -- completion TTFT ---------------------------------------------------------------

def test_completion_ttft_hand_built():
    """Two entries arrive at t=100 with work 30 and 50.  The drain window
    100..150 finishes the first at 130 (TTFT 30) and leaves 30 of the second,
    which the window 150..200 finishes at 180 (TTFT 80)."""
    o = O.Oracle(block_tokens=16, route_prefix_blocks=4, vnodes_per_instance=4, max_instances=4,
                 cache_capacity_blocks=64, slo_us=60, cost_us_per_token=1, hot_num=3, hot_den=2,
                 max_batch=8, max_batch_tokens=1 << 16, seed=1)
    assert o.add_instance(0) == 0 and o.add_instance(1) == 0
    assert o.route_batch([], [], [], 100)[0] == 0
    o.debug_enqueue(0, 0, 100, 0, 1, 0, 0, 30)
    o.debug_enqueue(0, 1, 100, 0, 1, 0, 0, 50)
    assert o.route_batch([], [], [], 150)[0] == 0
    m, _ = o.metrics()
    assert (m["completed"], m["ttft_sum_us"], m["ttft_max_us"], m["slo_met"]) == (1, 30, 30, 1)
    assert o.route_batch([], [], [], 200)[0] == 0
    m, hist = o.metrics()
    assert (m["completed"], m["ttft_sum_us"], m["ttft_max_us"], m["slo_met"]) == (2, 110, 80, 1)
    # p50 = rank 1 = 30, p90 = p99 = rank 2 = 80; both are bucket edges
    assert (m["ttft_p50_us"], m["ttft_p90_us"], m["ttft_p99_us"]) == (30, 80, 80)
    assert hist.sum() == 2 and hist[O.hist_bucket(30)] == 1 and hist[O.hist_bucket(80)] == 1
    assert m["requests"] == 0 and m["cv_samples"] == 0      # empty batches route nothing
    m, _ = o.metrics(reset=True)
    m, hist = o.metrics()
    assert m["completed"] == 0 and hist.sum() == 0


def test_completion_after_idle_gap():
    """An entry that arrives at an idle instance starts at its own arrival:
    routed at t=1000 with work 100 (100 uncached tokens, cost 1), it finishes
    at 1100 however long the next gap is."""
    o = O.Oracle(block_tokens=16, route_prefix_blocks=4, vnodes_per_instance=4, max_instances=4,
                 cache_capacity_blocks=64, slo_us=1000, cost_us_per_token=1, hot_num=3, hot_den=2,
                 max_batch=8, max_batch_tokens=1 << 16, seed=1)
    assert o.add_instance(0) == 0 and o.add_instance(1) == 0
    tok = np.arange(100, dtype=np.uint32)
    assert o.route_batch(tok, [0], [100], 1000)[0] == 0
    assert o.route_batch([], [], [], 5000)[0] == 0
    m, _ = o.metrics()
    assert (m["completed"], m["ttft_sum_us"], m["requests"], m["prompt_tokens"]) == (1, 100, 1, 100)
    assert m["est_slo_met"] == 1 and m["cv_samples"] == 1
    # after the one batch: W = [100, 0] (or mirrored): CV = |a-b|/(a+b) = 1
    assert m["cv_last"] == 1.0


# -- load CV and counters on a trace -------------------------------------------------

def _replay(rule, w, nb=None, check_cv=False):
    tr = Trace(w)
    o = O.Oracle(**O.config_from_workload(w, max_instances=w["n_instances"] + 4), choice_rule=rule)
    for i in range(w["n_instances"]):
        assert o.add_instance(i) == 0
    tot = dict(requests=0, prompt_tokens=0, hit_tokens=0, switched=0, est=0)
    cvs = []
    for b in range(len(tr.batches) if nb is None else nb):
        s, e, off, lens, ntok = tr.batch_layout(b)
        rc, out = o.route_batch(tr.batch_tokens(b), off, lens, tr.batch_time(b))
        assert rc == 0
        assert o.commit() == 0
        hch = np.where(out["chosen"] == out["cand1"], out["hit1"], out["hit2"])
        tch = np.where(out["chosen"] == out["cand1"], out["ttft1"], out["ttft2"])
        tot["requests"] += len(lens)
        tot["prompt_tokens"] += int(np.sum(lens))
        tot["hit_tokens"] += int(hch.sum())
        tot["switched"] += int(out["switched"].sum())
        if rule < GAFF:
            tot["est"] += int((tch <= w["slo_us"]).sum())
        if check_cv:
            W = o.loads()[o.inst_state() == 1].astype(np.float64)
            cv = W.std() / W.mean() if W.sum() else 0.0
            m, _ = o.metrics()
            assert m["cv_last"] == pytest.approx(cv, rel=1e-12, abs=1e-15)
            cvs.append(m["cv_last"])
    m, hist = o.metrics()
    assert m["requests"] == tot["requests"] and m["prompt_tokens"] == tot["prompt_tokens"]
    assert m["switched"] == tot["switched"]
    if rule <= GAFF:   # the chosen instance is one of the two candidates
        assert m["hit_tokens"] == tot["hit_tokens"]
    if rule < GAFF:
        assert m["est_slo_met"] == tot["est"]
    assert hist.sum() == m["completed"] <= m["requests"]
    if cvs:
        assert m["cv_sum"] == pytest.approx(sum(cvs), rel=1e-12)
    return m


@pytest.mark.parametrize("rule", ALL_RULES)
def test_counters_and_cv_against_numpy(rule):
    _replay(rule, workload("tiny", n_requests=600, batch=100), check_cv=True)


def test_rule_ordering_of_sec_2_2():
    """Sec. 2.2 on skewed shared prefixes, cluster-wide rules: cache affinity
    reaches the higher hit rate and least loaded the lower load imbalance
    (CV), with min TTFT and Preble between the two on both axes; DualMap
    keeps a hit rate comparable to cache affinity (Sec. 4.4) at a lower CV."""
    w = workload("tiny", n_requests=2000, batch=100, zipf_s=1.2, rho=0.9)
    res = {r: _replay(r, w) for r in (DM, GAFF, GLL, GMT, GPRE)}
    hit = {r: m["hit_tokens"] / m["prompt_tokens"] for r, m in res.items()}
    cv = {r: m["cv_sum"] / m["cv_samples"] for r, m in res.items()}
    assert hit[GAFF] > hit[GLL] and cv[GLL] < cv[GAFF]
    for r in (GMT, GPRE):
        assert hit[GLL] < hit[r] < hit[GAFF]
        assert cv[GLL] < cv[r] < cv[GAFF]
    assert hit[DM] >= 0.97 * hit[GAFF] and cv[DM] < cv[GAFF]


def test_completion_metrics_match_an_independent_queue_model():
    """Re-run the time model in plain Python from the oracle's routing
    decisions: one FIFO per instance, served at 1 us per us from each batch
    time; a request completes when the work ahead of it and its own is done.
    Its TTFT count, sum, max, SLO count, histogram and the estimated-SLO
    count must equal the oracle's metrics."""
    w = workload("tiny", n_requests=1500, batch=100, zipf_s=1.2, rho=1.1, slo_us=6000)
    tr = Trace(w)
    o = O.Oracle(**O.config_from_workload(w, max_instances=w["n_instances"]))
    for i in range(w["n_instances"]):
        assert o.add_instance(i) == 0
    cost, slo = w["cost_us"], w["slo_us"]
    queues = {i: [] for i in range(w["n_instances"])}   # [remaining, arrival]
    ttfts, est = [], 0
    t_prev = None
    for b in range(len(tr.batches)):
        s, e, off, lens, nt = tr.batch_layout(b)
        t = tr.batch_time(b)
        if t_prev is not None:                       # drain the window [t_prev, t)
            for q in queues.values():
                left, run = t - t_prev, 0
                while q and q[0][0] <= left - run:
                    rem, arr = q.pop(0)
                    run += rem
                    ttfts.append(t_prev + run - arr)
                if q:
                    q[0][0] -= left - run
        t_prev = t
        rc, out = o.route_batch(tr.batch_tokens(b), off, lens, t)
        assert rc == 0
        assert o.commit() == 0
        for r in range(len(lens)):
            ch = int(out["chosen"][r])
            h = int(out["hit1"][r] if ch == out["cand1"][r] else out["hit2"][r])
            queues[ch].append([cost * (int(lens[r]) - h), t])
            est += sum(x[0] for x in queues[ch]) <= slo
    m, hist = o.metrics()
    assert m["completed"] == len(ttfts) > 0
    assert m["ttft_sum_us"] == sum(ttfts) and m["ttft_max_us"] == max(ttfts)
    assert m["slo_met"] == sum(x <= slo for x in ttfts)
    assert m["est_slo_met"] == est
    want = np.zeros(O.HIST_BUCKETS, np.uint64)
    for x in ttfts:
        want[O.hist_bucket(x)] += 1
    assert np.array_equal(hist, want)
    srt = sorted(ttfts)
    for key, p in (("ttft_p50_us", 50), ("ttft_p90_us", 90), ("ttft_p99_us", 99)):
        exact = srt[max(1, -(-p * len(srt) // 100)) - 1]   # the ceil(p n)-th smallest
        assert m[key] == O.hist_lower(O.hist_bucket(exact))
        assert m[key] <= exact and (exact - m[key]) * 16 <= max(m[key], 16)


@pytest.mark.parametrize("rule", [GLL, GMT, GPRE])
def test_cluster_wide_rules_match_an_independent_model(rule):
    """Each request's choice under a cluster-wide rule, recomputed in plain
    Python: hits from the resident key sets as of the batch start (leading
    run of the prompt's block keys), loads from an independent FIFO model,
    then the rule's argmin in arrival order."""
    w = workload("tiny", n_requests=600, batch=100, zipf_s=1.2, rho=1.0)
    tr = Trace(w)
    n_inst, B, cost = w["n_instances"], w["block_tokens"], w["cost_us"]
    o = O.Oracle(**O.config_from_workload(w, max_instances=n_inst), choice_rule=rule)
    for i in range(n_inst):
        assert o.add_instance(i) == 0
    queues = {i: [] for i in range(n_inst)}
    t_prev = None
    for b in range(len(tr.batches)):
        s, e, off, lens, nt = tr.batch_layout(b)
        t = tr.batch_time(b)
        if t_prev is not None:
            for q in queues.values():
                left = t - t_prev
                while q and q[0] <= left:
                    left -= q.pop(0)
                if q:
                    q[0] -= left
        t_prev = t
        resident = {i: set(o.cache(i)[0].tolist()) for i in range(n_inst)}
        W = {i: sum(queues[i]) for i in range(n_inst)}
        tok = tr.batch_tokens(b)
        rc, out = o.route_batch(tok, off, lens, t)
        assert rc == 0
        for r in range(len(lens)):
            L = int(lens[r])
            keys = o.prompt_keys(tok[int(off[r]):int(off[r]) + L])[0].tolist()
            hits = {}
            for i in range(n_inst):
                m = 0
                while m < len(keys) and keys[m] in resident[i]:
                    m += 1
                hits[i] = B * m
            hmax = max(hits.values())
            if rule == GLL:
                key = {i: (W[i], i) for i in range(n_inst)}
            elif rule == GPRE and 2 * hmax > L:
                key = {i: (W[i], i) for i in range(n_inst) if hits[i] == hmax}
            else:
                key = {i: (W[i] + cost * (L - hits[i]), i) for i in range(n_inst)}
            ch = min(key, key=lambda i: key[i])
            assert int(out["chosen"][r]) == ch, (b, r)
            work = cost * (L - hits[ch])
            queues[ch].append(work)
            W[ch] += work
        assert o.commit() == 0


def _pair_choice(rule, c1, c2, h1, h2, L, W1, W2, slo, cost):
    """The two-candidate rules written out again in Python."""
    t1, t2 = W1 + cost * (L - h1), W2 + cost * (L - h2)
    if rule == DM:
        if h1 == h2:
            return c2 if W2 < W1 else c1
        a, b, Wa, Wb, ta = (c1, c2, W1, W2, t1) if h1 > h2 else (c2, c1, W2, W1, t2)
        if ta <= slo:
            return a
        return b if Wb < Wa else a
    if rule == AFF or (rule == PRE and 2 * max(h1, h2) > L):
        if h1 != h2:
            return c1 if h1 > h2 else c2
        return c2 if W2 < W1 else c1
    if rule == LL:
        return c2 if W2 < W1 else c1
    return c2 if t2 < t1 else c1                       # min TTFT, and Preble below half


@pytest.mark.parametrize("rule", [DM, AFF, LL, MT, PRE])
def test_pair_rules_match_an_independent_model_on_a_trace(rule):
    """DualMap's rule and the pair variants on a trace under load (the SLO
    switch fires): loads from an independent FIFO model, the reported
    candidates and hits, each choice recomputed in arrival order."""
    w = workload("tiny", n_requests=1000, batch=100, zipf_s=1.2, rho=1.2, slo_us=3000)
    tr = Trace(w)
    n_inst, cost, slo = w["n_instances"], w["cost_us"], w["slo_us"]
    o = O.Oracle(**O.config_from_workload(w, max_instances=n_inst), choice_rule=rule)
    for i in range(n_inst):
        assert o.add_instance(i) == 0
    queues = {i: [] for i in range(n_inst)}
    t_prev, switched = None, 0
    for b in range(len(tr.batches)):
        s, e, off, lens, nt = tr.batch_layout(b)
        t = tr.batch_time(b)
        if t_prev is not None:
            for q in queues.values():
                left = t - t_prev
                while q and q[0] <= left:
                    left -= q.pop(0)
                if q:
                    q[0] -= left
        t_prev = t
        W = {i: sum(queues[i]) for i in range(n_inst)}
        rc, out = o.route_batch(tr.batch_tokens(b), off, lens, t)
        assert rc == 0
        for r in range(len(lens)):
            c1, c2 = int(out["cand1"][r]), int(out["cand2"][r])
            h1, h2, L = int(out["hit1"][r]), int(out["hit2"][r]), int(lens[r])
            ch = _pair_choice(rule, c1, c2, h1, h2, L, W[c1], W[c2], slo, cost)
            assert int(out["chosen"][r]) == ch, (b, r)
            assert int(out["ttft1"][r]) == W[c1] + cost * (L - h1)
            work = cost * (L - (h1 if ch == c1 else h2))
            queues[ch].append(work)
            W[ch] += work
        switched += int(out["switched"].sum())
        assert o.commit() == 0
    if rule == DM:
        assert switched > 0


def test_cv_counts_live_instances_only():
    """A removed instance keeps draining its queue but is not part of the
    cluster whose balance the CV measures (Sec. 2.2: the instances serving
    requests): its queued work is left out of the sample."""
    w = workload("tiny", n_requests=400, batch=100)
    tr = Trace(w)
    o = O.Oracle(**O.config_from_workload(w, max_instances=w["n_instances"]))
    for i in range(w["n_instances"]):
        assert o.add_instance(i) == 0
    for b in range(2):
        s, e, off, lens, nt = tr.batch_layout(b)
        assert o.route_batch(tr.batch_tokens(b), off, lens, tr.batch_time(b))[0] == 0
        assert o.commit() == 0
    gone = int(np.argmax(o.loads()))
    assert o.loads()[gone] > 0 and o.remove_instance(gone) == 0
    s, e, off, lens, nt = tr.batch_layout(2)
    assert o.route_batch(tr.batch_tokens(2), off, lens, tr.batch_time(1))[0] == 0   # no time passes
    m, _ = o.metrics()
    W = o.loads().astype(np.float64)
    live = o.inst_state() == 1
    assert not live[gone] and W[gone] > 0
    assert m["cv_last"] == pytest.approx(W[live].std() / W[live].mean(), rel=1e-12)
    assert m["cv_last"] != pytest.approx(W.std() / W.mean(), rel=1e-6)
