"""Bit-exact parity of the CUDA routing path (through the C ABI) with the CPU
oracle on seeded synthetic traces of all five workload shapes, plus edge
cases and error behaviour."""

import numpy as np
import pytest

from parity_harness import Pair, lib_ready, run_trace
from tracegen import Trace, workload

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    lib_ready()


def _torch():
    import torch
    return torch


# -- inputs and hashing ------------------------------------------------------------

def test_device_token_filler_matches_host():
    torch = _torch()
    import tracegen.device as TD
    tr = Trace(workload("multiturn", n_requests=300, batch=100))
    r0, r1 = 37, 211
    n = int(tr.req_off[r1] - tr.req_off[r0])
    buf = torch.zeros(n + 4, dtype=torch.int32, device="cuda")
    TD.fill_range(tr, r0, r1, buf)
    got = buf.cpu().numpy().view(np.uint32)
    for r in range(r0, r1):
        o = int(tr.req_off[r] - tr.req_off[r0])
        assert np.array_equal(got[o:o + tr.L[r]], tr.request_tokens(r)), r


def _lengths_mix(B, rng):
    """Edge lengths (exactly one block, one block + 1, segment boundaries of
    256 blocks, a ragged tail) plus random lengths spanning several segments."""
    fixed = [B, B + 1, 2 * B - 1, 31 * B, 32 * B, 33 * B + 3, 256 * B, 256 * B + 1, 257 * B, 600 * B + 5]
    return fixed + rng.integers(B, 900 * B, size=40).tolist()


@pytest.mark.parametrize("B,K", [(16, 16), (4, 1), (8, 40), (32, 7), (64, 256), (16, 256)])
def test_hash_prompts_parity(B, K):
    torch = _torch()
    from oracle import oracle as O
    from paper_2602_06502_gb300 import dualmap as D
    from paper_2602_06502_gb300.scheduler import Scheduler
    rng = np.random.default_rng(B * 1000 + K)
    lens = np.array(_lengths_mix(B, rng), np.uint32)
    off = np.zeros(len(lens), np.uint64)
    off[1:] = np.cumsum((lens[:-1] + 3) // 4 * 4)
    ntok = int(off[-1] + lens[-1])
    tok = rng.integers(0, 1 << 32, size=ntok, dtype=np.uint64).astype(np.uint32)
    seed = 77 + B
    ora = O.Oracle(block_tokens=B, route_prefix_blocks=K, vnodes_per_instance=4, max_instances=4,
                   cache_capacity_blocks=16, slo_us=1, cost_us_per_token=1, hot_num=3, hot_den=2,
                   max_batch=len(lens), max_batch_tokens=1 << 24, seed=seed)
    g = Scheduler(block_tokens=B, route_prefix_blocks=K, vnodes=4, max_instances=4, capacity=16,
                  max_batch=len(lens), max_batch_tokens=ntok + 64, seed=seed)
    dt = torch.from_numpy(tok.view(np.int32)).cuda()
    do = torch.from_numpy(off.view(np.int64)).cuda()
    dl = torch.from_numpy(lens.view(np.int32)).cuda()
    nblk = lens // B
    keys = torch.zeros(int(nblk.sum()) + 1, dtype=torch.int64, device="cuda")
    koff = torch.zeros(len(lens) + 1, dtype=torch.int64, device="cuda")
    pos = torch.zeros(2 * len(lens), dtype=torch.int64, device="cuda")
    b = D.make_batch(dt, do, dl, len(lens), ntok, 0)
    assert D.dm_hash_prompts(g.h, b, keys, koff, pos) == 0
    assert g.last_error() == 0
    keys = keys.cpu().numpy().view(np.uint64)
    koff = koff.cpu().numpy().view(np.uint64)
    pos = pos.cpu().numpy().view(np.uint64).reshape(-1, 2)
    assert np.array_equal(np.diff(koff.astype(np.int64)), nblk.astype(np.int64))
    for r in range(len(lens)):
        want_k, want_p = ora.prompt_keys(tok[int(off[r]):int(off[r]) + int(lens[r])])
        got_k = keys[int(koff[r]):int(koff[r + 1])]
        assert np.array_equal(got_k, want_k), (r, int(lens[r]))
        assert np.array_equal(pos[r], want_p), r
    g.close()


def test_ring_parity_add_remove_lookup():
    torch = _torch()
    from oracle import oracle as O
    from paper_2602_06502_gb300 import dualmap as D
    w = workload("tiny", vnodes=37)
    p = Pair(w, max_instances=20)
    rng = np.random.default_rng(4)
    pos = rng.integers(0, 2**63, size=2000, dtype=np.int64).astype(np.uint64) * np.uint64(2)

    def check():
        for f in (0, 1):
            vp, ow, _ = p.ora.ring(f)
            gv, go = D.dm_export_ring(p.gpu.h, f, len(vp) + 8)
            assert np.array_equal(gv, vp) and np.array_equal(go, ow)
        dpos = torch.from_numpy(pos.view(np.int64)).cuda()
        o1 = torch.zeros(len(pos) // 2, dtype=torch.int32, device="cuda")
        o2 = torch.zeros_like(o1)
        assert D.dm_ring_lookup(p.gpu.h, dpos, len(pos) // 2, o1, o2) == 0
        pr = pos.reshape(-1, 2)
        assert np.array_equal(o1.cpu().numpy().astype(np.uint32), p.ora.ring_owners(pr[:, 0].copy(), 0))
        assert np.array_equal(o2.cpu().numpy().astype(np.uint32), p.ora.ring_owners(pr[:, 1].copy(), 1))
        # a position equal to a vnode position belongs to that vnode
        vp, ow, _ = p.ora.ring(0)
        m = min(200, len(vp))
        eq = np.repeat(vp[:m], 2)
        deq = torch.from_numpy(eq.view(np.int64)).cuda()
        assert D.dm_ring_lookup(p.gpu.h, deq, m, o1, o2) == 0
        assert np.array_equal(o1[:m].cpu().numpy().astype(np.uint32), ow[:m])

    for i in [0, 3, 1, 7]:
        p.add(i)
        check()
    for i in range(8, 20):
        p.add(i)
    check()
    for i in [3, 19, 8, 0]:
        p.remove(i)
        check()
    p.add(19)   # removed, nothing queued: may be re-added
    check()


# -- whole traces -------------------------------------------------------------------

@pytest.mark.parametrize("seed", [1001, 1, 2, 3, 4, 5, 6])
def test_tiny_trace_parity(seed):
    tr = Trace(workload("tiny"), seed=seed)
    run_trace(Pair(tr.cfg), tr, state_every=4)


def test_tiny_trace_with_rebalance_and_small_cache():
    """Eviction every batch, log compaction and index rebuilds (small C and
    touch bound), rebalancing after every batch: commits whose plan must
    recount the blocks per instance because a rebalance moved a request of
    the batch meet commits that compact or rebuild."""
    from paper_2602_06502_gb300 import dualmap as D
    w = workload("tiny", n_requests=2000, batch=100, capacity=700, zipf_s=1.3, rho=1.2)
    tr = Trace(w)
    p = Pair(w, max_touch=2600)
    run_trace(p, tr, rebalance=True, state_every=5)
    rebuilds, compactions = D.dm_get_maint_counts(p.gpu.h)
    print(f"{p.n_migrations} migrations, {rebuilds} index rebuilds, {compactions} log compactions")
    assert p.n_migrations > 0 and rebuilds + compactions > 0


def test_multiturn_parity():
    tr = Trace(workload("multiturn", n_requests=6144))
    p = Pair(tr.cfg, max_batch_tokens=1 << 25, capacity=60_000, max_touch=200_000)
    run_trace(p, tr, state_every=3)


def test_agent_parity():
    tr = Trace(workload("agent", n_requests=3 * 4096))
    p = Pair(tr.cfg, max_batch_tokens=40_000_000, max_touch=1 << 20)
    run_trace(p, tr)
    assert p.n_switched > 0      # the tight load makes the SLO rule fire


def test_longctx_parity():
    tr = Trace(workload("longctx", n_requests=3 * 512))
    p = Pair(tr.cfg, max_batch_tokens=70_000_000, max_touch=1 << 20, capacity=200_000)
    run_trace(p, tr)


def test_scaling_parity_with_events():
    """256 instances x 1,024 vnodes, rebalancing after every batch, an instance
    added or removed between batches."""
    w = workload("scaling", n_requests=5 * 4096, scale_every=4096, capacity=20_000)
    tr = Trace(w)
    assert len(tr.events) >= 3
    p = Pair(tr.cfg, max_instances=w["n_instances"] + 4, max_batch_tokens=40_000_000, max_touch=1 << 20)
    run_trace(p, tr, rebalance=True)


# -- choice rules and serving metrics -------------------------------------------------

RULES = list(range(9))   # dm_choice_rule: DualMap, four pair variants, four cluster-wide rules


@pytest.mark.parametrize("rule", RULES)
def test_choice_rules_tiny(rule):
    """Every rule, bit for bit, with the metrics (completion TTFTs, CV)."""
    w = workload("tiny", n_requests=2000, batch=100, zipf_s=1.2, rho=0.9, slo_us=20_000)
    tr = Trace(w)
    m = run_trace(Pair(w, choice_rule=rule), tr, state_every=5)
    assert m["requests"] == 2000 and m["completed"] > 0 and m["cv_samples"] == 20


@pytest.mark.parametrize("rule", [0, 3, 7, 8])
def test_choice_rules_agent(rule):
    """Tight load (the SLO switch fires), 64 instances, 4,096-request batches."""
    tr = Trace(workload("agent", n_requests=2 * 4096))
    p = Pair(tr.cfg, max_batch_tokens=40_000_000, max_touch=1 << 20, choice_rule=rule)
    run_trace(p, tr)


@pytest.mark.parametrize("rule", [0, 6, 8])
def test_choice_rules_with_scaling_and_rebalance(rule):
    """Instances added and removed between batches (the cluster-wide rules
    skip removed ones), rebalancing after every batch (migrated requests
    keep their arrival time for the TTFT)."""
    w = workload("scaling", n_requests=4 * 2048, batch=2048, scale_every=2048, n_instances=48, vnodes=64,
                 capacity=20_000)
    tr = Trace(w)
    assert len(tr.events) >= 3
    p = Pair(tr.cfg, max_instances=w["n_instances"] + 4, max_batch_tokens=20_000_000, max_touch=1 << 20,
             choice_rule=rule)
    run_trace(p, tr, rebalance=True)


def test_metrics_reset_and_rebalanced_ttft():
    """Completion TTFTs after migrations, then a reset clears every metric."""
    from paper_2602_06502_gb300 import dualmap as D
    w = workload("tiny", n_requests=1500, batch=100, capacity=700, zipf_s=1.3, rho=1.2)
    tr = Trace(w)
    p = Pair(w, max_touch=2600)
    run_trace(p, tr, rebalance=True)
    assert p.n_migrations > 0
    gm, gh = D.dm_get_metrics(p.gpu.h, reset=True)
    assert gm["completed"] > 0
    gm, gh = D.dm_get_metrics(p.gpu.h)
    assert all(v == 0 for v in gm.values()) and gh.sum() == 0


# -- adaptive hash-prefix length --------------------------------------------------------

def _ad(step, kmax, window=1):
    return dict(adapt_step_blocks=step, adapt_max_blocks=kmax, adapt_window=window)


@pytest.mark.parametrize("window", [1, 2])
def test_adaptive_prefix_tiny(window):
    """Zipf-1.2 prefixes over 8 instances: the top prefixes pass 2/n and
    deepen 8 blocks per window up to their shared length; every request's
    length and the expanded nodes match the oracle after every batch."""
    w = workload("tiny", n_requests=2000, batch=100, zipf_s=1.2, rho=0.9)
    tr = Trace(w)
    p = Pair(w, adapt=_ad(8, 128, window))
    run_trace(p, tr, state_every=5)
    from paper_2602_06502_gb300 import dualmap as D
    assert len(D.dm_export_prefix_tree(p.gpu.h)) > 0


def test_adaptive_prefix_agent():
    tr = Trace(workload("agent", n_requests=3 * 4096))
    p = Pair(tr.cfg, max_batch_tokens=40_000_000, max_touch=1 << 20, adapt=_ad(32, 1024))
    run_trace(p, tr)


def test_adaptive_prefix_longctx_deepens_past_shared_prefix():
    """16k-token shared prefixes (1,024 blocks), 128 instances: hot prefixes
    deepen 128 blocks per batch; the longest lengths grow batch by batch."""
    tr = Trace(workload("longctx", n_requests=6 * 512))
    p = Pair(tr.cfg, max_batch_tokens=70_000_000, max_touch=1 << 20, capacity=200_000, adapt=_ad(128, 2048))
    run_trace(p, tr)
    assert int(p.ora.route_blocks().max()) > 16 + 3 * 128


def test_adaptive_prefix_with_scaling_and_rebalance():
    w = workload("scaling", n_requests=4 * 2048, batch=2048, scale_every=2048, n_instances=48, vnodes=64,
                 capacity=20_000)
    tr = Trace(w)
    p = Pair(tr.cfg, max_instances=w["n_instances"] + 4, max_batch_tokens=20_000_000, max_touch=1 << 20,
             adapt=_ad(16, 256))
    run_trace(p, tr, rebalance=True)


# -- rebalancing variants -------------------------------------------------------------

@pytest.mark.parametrize("flags", [0, 1, 2, 3])
def test_rebalance_variants_skewed(flags):
    """A skewed 16-instance workload with a 5 ms SLO, rebalancing after every
    batch: the 1.5x-mean rule, the SLO target, the double-overload trigger
    and both (DM_REBALANCE_* bits); migrations bit for bit."""
    w = workload("scaling", n_requests=3000, batch=50, n_instances=16, vnodes=32, n_prefix=100, zipf_s=1.2,
                 len_lo=400, len_hi=512, prefix_lo=384, prefix_hi=384, scale_every=0, rho=1.0, slo_us=5000)
    tr = Trace(w)
    p = Pair(w, max_instances=16, rebalance_flags=flags)
    run_trace(p, tr, rebalance=True, state_every=10)
    assert p.n_migrations > 0


@pytest.mark.parametrize("flags", [1, 3])
def test_rebalance_variants_tiny(flags):
    w = workload("tiny", n_requests=2000, batch=100, capacity=700, zipf_s=1.3, rho=1.2, slo_us=20_000)
    tr = Trace(w)
    p = Pair(w, max_touch=2600, rebalance_flags=flags)
    run_trace(p, tr, rebalance=True, state_every=5)
    assert p.n_migrations > 0


@pytest.mark.parametrize("flags", [4, 5, 7])
def test_rebalance_fresh_hits(flags):
    """DM_REBALANCE_FRESH_HITS (with the SLO target, and with both other
    variants): every migration candidate's hit on its other candidate is
    probed afresh from its keys in the per-instance key rings; migrations,
    loads, queues and resident keys bit for bit with the oracle, on the
    skewed workload (where fresh and stored hits differ) and on a small-cache
    tiny trace with evictions between the routing and the rebalance of
    requests queued earlier."""
    w = workload("scaling", n_requests=3000, batch=50, n_instances=16, vnodes=32, n_prefix=100, zipf_s=1.2,
                 len_lo=400, len_hi=512, prefix_lo=384, prefix_hi=384, scale_every=0, rho=1.0, slo_us=5000)
    p = Pair(w, max_instances=16, rebalance_flags=flags, rebalance_key_blocks=1 << 16)
    run_trace(p, Trace(w), rebalance=True, state_every=10)
    assert p.n_migrations > 0
    w = workload("tiny", n_requests=2000, batch=100, capacity=700, zipf_s=1.3, rho=1.2, slo_us=20_000)
    p = Pair(w, max_touch=2600, rebalance_flags=flags, rebalance_key_blocks=1 << 16)
    run_trace(p, Trace(w), rebalance=True, state_every=5)


def test_rebalance_fresh_hits_change_migrations():
    """On a skewed workload at rho 1.2 with a 20 ms SLO the fresh hits change
    which requests move (the oracle shows it); the GPU's fresh-hit run is in
    parity with the oracle call by call.  A key ring too small for the
    queued requests' keys is a sticky DM_ERR_CAPACITY, not a silent
    overwrite."""
    from oracle import oracle as O
    from paper_2602_06502_gb300 import dualmap as D
    w = workload("scaling", n_requests=3000, batch=50, n_instances=16, vnodes=32, n_prefix=100, zipf_s=1.2,
                 len_lo=400, len_hi=512, prefix_lo=384, prefix_hi=384, scale_every=0, rho=1.2, slo_us=20000)
    tr = Trace(w)
    lists = {}
    for flags in (0, O.RB_FRESH_HITS):
        o = O.Oracle(**O.config_from_workload(w, max_instances=16), rebalance_flags=flags)
        for i in range(16):
            assert o.add_instance(i) == 0
        got = []
        for b in range(len(tr.batches)):
            s, e, off, lens, nt = tr.batch_layout(b)
            assert o.route_batch(tr.batch_tokens(b), off, lens, tr.batch_time(b))[0] == 0
            rc, n, (seq, fr, to) = o.rebalance()
            got += list(zip(seq.tolist(), fr.tolist(), to.tolist()))
            assert o.commit() == 0
        lists[flags] = got
    assert lists[0] != lists[O.RB_FRESH_HITS]
    p = Pair(w, max_instances=16, rebalance_flags=D.DM_REBALANCE_FRESH_HITS, rebalance_key_blocks=1 << 16)
    run_trace(p, tr, rebalance=True, state_every=10)
    assert p.n_migrations == len(lists[O.RB_FRESH_HITS])
    from paper_2602_06502_gb300.scheduler import Scheduler
    g = Scheduler(block_tokens=16, route_prefix_blocks=16, vnodes=32, max_instances=16, capacity=4096, slo_us=5000,
                  max_batch=64, max_batch_tokens=1 << 16, rebalance_flags=D.DM_REBALANCE_FRESH_HITS,
                  rebalance_key_blocks=64)
    for i in range(4):
        assert g.add_instance(i) == 0
    import torch
    tr = Trace(w)
    s, e, off, lens, nt = tr.batch_layout(0)
    dev = torch.device("cuda:0")
    tok = torch.from_numpy(tr.batch_tokens(0).view(np.int32)).to(dev)
    g.route(tok, torch.from_numpy(off.view(np.int64)).to(dev), torch.from_numpy(lens.view(np.int32)).to(dev),
            e - s, nt, tr.batch_time(0), check=False)
    assert g.last_error() == D.DM_ERR_CAPACITY      # 50 prompts of ~28 blocks on 4 instances: over 64 per ring


def test_rebalance_fresh_hits_arguments():
    from paper_2602_06502_gb300 import dualmap as D
    from paper_2602_06502_gb300.scheduler import Scheduler
    for kw in (dict(rebalance_key_blocks=0), dict(rebalance_key_blocks=1024, choice_rule=D.DM_RULE_MIN_TTFT),
               dict(rebalance_key_blocks=1024, candidates=3)):
        with pytest.raises(D.DualMapError):
            Scheduler(max_instances=8, rebalance_flags=D.DM_REBALANCE_FRESH_HITS, **kw)


# -- features combined ------------------------------------------------------------------

@pytest.mark.parametrize("rule,flags", [(7, 3), (3, 1)])
def test_rule_adaptive_and_rebalance_together(rule, flags):
    """A compared rule, the adaptive hash length and a rebalancing variant in
    one run: they share the route, choice and rebalance kernels' state."""
    w = workload("scaling", n_requests=3000, batch=50, n_instances=16, vnodes=32, n_prefix=100, zipf_s=1.2,
                 len_lo=400, len_hi=512, prefix_lo=384, prefix_hi=384, scale_every=0, rho=1.0, slo_us=5000)
    tr = Trace(w)
    p = Pair(w, max_instances=16, choice_rule=rule, rebalance_flags=flags, adapt=_ad(4, 32))
    run_trace(p, tr, rebalance=True, state_every=10)
    from paper_2602_06502_gb300 import dualmap as D
    assert len(D.dm_export_prefix_tree(p.gpu.h)) > 0


# -- edge cases ---------------------------------------------------------------------

def _mk(**kw):
    base = dict(workload("tiny"))
    base.update(kw)
    return base


def _batch(prompts):
    lens = np.array([len(x) for x in prompts], np.uint32)
    off = np.zeros(len(prompts), np.uint64)
    if len(prompts) > 1:
        off[1:] = np.cumsum((lens[:-1].astype(np.uint64) + 3) // 4 * 4)
    tot = int(off[-1] + lens[-1]) if len(prompts) else 0
    tok = np.zeros(max(tot, 4), np.uint32)
    for o, x in zip(off, prompts):
        tok[int(o):int(o) + len(x)] = x
    return tok, off, lens


def test_edge_cases_small_clusters():
    rng = np.random.default_rng(12)
    w = _mk(n_instances=2, vnodes=1, capacity=50, batch=64)
    p = Pair(w, max_instances=3)
    p.add(0)
    p.add(1)
    same = rng.integers(0, 32000, size=16 * 9, dtype=np.uint32)
    t = 0
    for step in range(6):
        prompts = [same] * 5 + [rng.integers(0, 32000, size=int(L), dtype=np.uint32)
                                for L in (16, 17, 31, 32, 48, 16 * 64)]
        tok, off, lens = _batch(prompts)
        p.route(tok, off, lens, t, tag=f"step {step}")
        p.rebalance()
        p.commit()
        p.check_state()
        t += 7
    # a batch of one, then an empty batch (time only), then identical time
    tok, off, lens = _batch([same])
    p.route(tok, off, lens, t)
    p.commit()
    p.route(np.zeros(4, np.uint32), np.zeros(0, np.uint64), np.zeros(0, np.uint32), t + 100)
    p.commit()
    p.check_state()
    p.add(2)
    p.remove(0)            # remove down to two live instances
    tok, off, lens = _batch([same] * 3)
    p.route(tok, off, lens, t + 100)
    p.commit()
    p.check_state()


def test_zero_load_and_non_dense_ids():
    rng = np.random.default_rng(13)
    w = _mk(vnodes=16, capacity=10_000, batch=128)
    p = Pair(w, max_instances=12)
    for i in (1, 4, 5, 9, 11):
        p.add(i)
    prompts = [rng.integers(0, 32000, size=int(L), dtype=np.uint32) for L in rng.integers(16, 3000, size=100)]
    tok, off, lens = _batch(prompts)
    p.route(tok, off, lens, 0)             # W = 0 everywhere at the start
    p.commit()
    p.remove(5)
    p.route(tok, off, lens, 10**9)          # everything drained: W = 0 again
    p.rebalance()
    p.commit()
    p.check_state()


def test_error_statuses_match_oracle():
    from paper_2602_06502_gb300 import dualmap as D
    rng = np.random.default_rng(14)
    w = _mk(batch=4)
    p = Pair(w, max_instances=6)
    tok, off, lens = _batch([rng.integers(0, 32000, size=64, dtype=np.uint32)])
    dt, do, dl = p.to_dev(tok, off, lens)
    assert p.gpu.route(dt, do, dl, 1, len(tok), 0, check=False) == D.DM_ERR_NO_INSTANCES
    assert p.add(0) == 0
    assert p.add(0) == D.DM_ERR_DUPLICATE_ID
    assert p.add(6) == D.DM_ERR_INVALID_ARG
    assert p.remove(3) == D.DM_ERR_UNKNOWN_ID
    assert p.add(1) == 0
    p.route(tok, off, lens, 50)
    assert p.gpu.route(dt, do, dl, 1, len(tok), 49, check=False) == D.DM_ERR_ORDER
    assert p.ora.route_batch(tok, off, lens, 49)[0] == D.DM_ERR_ORDER
    tok5, off5, lens5 = _batch([tok[:16]] * 5)
    d5 = p.to_dev(tok5, off5, lens5)
    assert p.gpu.route(*d5, 5, len(tok5), 60, check=False) == D.DM_ERR_CAPACITY
    # a removed instance with queued work cannot come back until drained
    busy = int(p.gpu.results(1)["chosen"][0])
    assert p.remove(busy) == 0
    assert p.add(busy) == D.DM_ERR_DUPLICATE_ID
    assert p.gpu.last_error() == 0


def test_device_side_validation_is_sticky():
    """A prompt shorter than one block is rejected in the set-up kernel: the
    call's kernels do nothing and the handle reports the error."""
    torch = _torch()
    from paper_2602_06502_gb300 import dualmap as D
    from paper_2602_06502_gb300.scheduler import Scheduler
    g = Scheduler(vnodes=8, max_instances=4, max_batch=4, max_batch_tokens=1 << 12, seed=3)
    g.add_instance(0)
    g.add_instance(1)
    tok = torch.zeros(64, dtype=torch.int32, device="cuda")
    off = torch.tensor([0, 16], dtype=torch.int64, device="cuda")
    ln = torch.tensor([32, 15], dtype=torch.int32, device="cuda")
    assert g.route(tok, off, ln, 2, 64, 0, check=False) == 0
    assert g.last_error() == D.DM_ERR_INVALID_ARG
    assert np.all(g.loads() == 0)                 # nothing was queued
    assert g.route(tok, off, ln, 2, 64, 1, check=False) == D.DM_ERR_INVALID_ARG
    g.close()
    g = Scheduler(vnodes=8, max_instances=4, max_batch=4, max_batch_tokens=1 << 12, seed=3)
    g.add_instance(0)
    g.add_instance(1)
    off = torch.tensor([0, 18], dtype=torch.int64, device="cuda")    # not 16-byte aligned
    ln = torch.tensor([16, 16], dtype=torch.int32, device="cuda")
    assert g.route(tok, off, ln, 2, 64, 0, check=False) == 0
    assert g.last_error() == D.DM_ERR_INVALID_ARG
    g.close()


def test_host_buffer_entry_point_matches_device_path():
    from paper_2602_06502_gb300 import dualmap as D
    from paper_2602_06502_gb300.scheduler import OUT_FIELDS
    tr = Trace(workload("tiny", n_requests=768, batch=256))
    a = Pair(tr.cfg)
    b = Pair(tr.cfg)
    for i in range(tr.cfg["n_instances"]):
        a.add(i)
        b.add(i)
    for k in range(len(tr.batches)):
        s, e, off, lens, ntok = tr.batch_layout(k)
        tok = tr.batch_tokens(k)
        want = a.route(tok, off, lens, tr.batch_time(k))
        n = e - s
        host = {name: np.zeros(n, dtype={"int32": np.uint32, "int64": np.uint64, "uint8": np.uint8}[str(t).split(".")[1]])
                for name, t in OUT_FIELDS}
        bt = D.make_batch(tok, off, lens, n, ntok, tr.batch_time(k))
        out = D.make_out(*[host[name] for name, _ in OUT_FIELDS])
        assert D.dm_route_batch_host(b.gpu.h, bt, out) == 0
        b.ora.route_batch(tok, off, lens, tr.batch_time(k))
        for name in want:
            assert np.array_equal(host[name], want[name]), name
        a.commit()
        b.commit()
    b.check_state()


def test_longctx_full_size_batches():
    """The long-context workload at its real sizes (512 prompts of 32k-131k
    tokens per batch) in the launch configuration the benchmark uses: the
    first batches compared in full."""
    from bench import longctx_handle_kwargs
    tr = Trace(workload("longctx"))
    kw = longctx_handle_kwargs(tr.cfg)
    p = Pair(tr.cfg, max_instances=kw["max_instances"], max_batch_tokens=kw["max_batch_tokens"],
             max_touch=kw["max_touch_per_instance"], index_slots_log2=kw["index_slots_log2"])
    run_trace(p, tr, batches=2, check_state_end=False)
    p.check_state(ids=range(0, 128, 9))


def test_host_async_pipeline_matches_oracle():
    """Asynchronous host-buffer routing: several batches enqueued back to back
    (uploads overlapping routing on the two staging buffers), one wait, every
    batch's results equal to the oracle's."""
    from paper_2602_06502_gb300 import dualmap as D
    from paper_2602_06502_gb300.scheduler import OUT_FIELDS
    import torch
    tr = Trace(workload("tiny", n_requests=1280, batch=256))
    p = Pair(tr.cfg)
    for i in range(tr.cfg["n_instances"]):
        p.add(i)
    npdt = {"int32": np.uint32, "int64": np.uint64, "uint8": np.uint8}
    keep, wants = [], []
    for k in range(len(tr.batches)):
        s, e, off, lens, ntok = tr.batch_layout(k)
        tok = tr.batch_tokens(k)
        rc, want = p.ora.route_batch(tok, off, lens, tr.batch_time(k))
        assert rc == 0 and p.ora.commit() == 0
        n = e - s
        pin = {"tok": torch.from_numpy(tok.view(np.int32)).pin_memory(),
               "off": torch.from_numpy(off.view(np.int64)).pin_memory(),
               "len": torch.from_numpy(lens.view(np.int32)).pin_memory()}
        host = {name: torch.zeros(n, dtype=t).pin_memory() for name, t in OUT_FIELDS}
        bt = D.make_batch(pin["tok"], pin["off"], pin["len"], n, ntok, tr.batch_time(k))
        assert D.dm_route_batch_host_async(p.gpu.h, bt, D.make_out(*[host[name] for name, _ in OUT_FIELDS])) == 0
        p.gpu.commit()
        keep.append((pin, host))
        wants.append(want)
    assert p.gpu.last_error() == 0
    for (pin, host), want in zip(keep, wants):
        for name, t in OUT_FIELDS:
            got = host[name].numpy().view(npdt[str(t).split(".")[1]])
            assert np.array_equal(got, want[name]), name
    p.check_state()


# -- index maintenance and placement stress ----------------------------------------

def _run_prompts(p, batches, t0=0, dt=10, rebalance=False, state_every=1):
    t = t0
    for k, prompts in enumerate(batches):
        tok, off, lens = _batch(prompts)
        p.route(tok, off, lens, t, tag=f"batch {k}")
        if rebalance:
            p.rebalance(tag=f"batch {k}")
        p.commit()
        p.check_loads(tag=f"batch {k}")
        if state_every and (k + 1) % state_every == 0:
            p.check_state(tag=f"batch {k}")
        t += dt
    return t


def test_index_rebuild_and_log_compaction():
    """Prompts that are only a few hot prefixes re-touch the same keys every
    batch: the log fills with stale records while nothing is evicted, until it
    must be compacted.  Batches of unique prompts then fill the index past
    half, forcing rebuilds.  Both paths stay bit-exact, and the maintenance
    counters show that each ran."""
    from paper_2602_06502_gb300 import dualmap as D
    rng = np.random.default_rng(21)
    w = _mk(n_instances=2, vnodes=16, capacity=1000, batch=64)
    p = Pair(w, max_instances=3, max_touch=4096)
    p.add(0)
    p.add(1)
    hot = [rng.integers(0, 32000, size=16 * 64, dtype=np.uint32) for _ in range(4)]
    batches = [[hot[int(i)] for i in rng.integers(0, 4, size=64)] for _ in range(12)]
    t = _run_prompts(p, batches, state_every=3)
    rebuilds0, compactions = D.dm_get_maint_counts(p.gpu.h)
    assert compactions >= 1, (rebuilds0, compactions)
    uniq = [[rng.integers(0, 32000, size=16 * 64, dtype=np.uint32) for _ in range(64)] for _ in range(8)]
    _run_prompts(p, uniq, t0=t, state_every=2)
    rebuilds, compactions2 = D.dm_get_maint_counts(p.gpu.h)
    assert rebuilds > rebuilds0, (rebuilds, compactions2)


def test_rebuilds_share_a_one_buffer_pool():
    """One spare index buffer for all instances: two instances filling their
    indices at the same rate cross half full together, so one rebuild waits
    a commit for the buffer the other returns; results stay bit-exact and
    the rebuild counter keeps rising."""
    from paper_2602_06502_gb300 import dualmap as D
    rng = np.random.default_rng(24)
    w = _mk(n_instances=3, vnodes=16, capacity=1000, batch=64)
    p = Pair(w, max_instances=3, max_touch=4096, index_slots_log2=15, rebuild_pool=1)
    for i in range(3):
        assert p.add(i) == 0
    uniq = [[rng.integers(0, 32000, size=16 * 64, dtype=np.uint32) for _ in range(64)] for _ in range(30)]
    t = _run_prompts(p, uniq[:24], state_every=3)
    rebuilds, _ = D.dm_get_maint_counts(p.gpu.h)
    assert rebuilds >= 3, rebuilds
    assert p.remove(1) == 0
    t = _run_prompts(p, uniq[24:26], t0=t + 10**9, state_every=1)   # instance 1's queue drains
    assert p.add(1) == 0                   # a re-added id keeps whichever buffer it holds now
    _run_prompts(p, uniq[26:], t0=t, state_every=1)


def test_eviction_of_more_than_one_round():
    """Each commit evicts about 327k records per instance, more than one
    eviction round covers (a round reads 32k-128k records: four CTAs of 512
    threads, 16-64 records each, sized to twice what is left to evict)."""
    rng = np.random.default_rng(22)
    w = _mk(n_instances=2, vnodes=16, capacity=1000, batch=80)
    p = Pair(w, max_instances=3, max_touch=1 << 20, max_batch_tokens=1 << 24)
    p.add(0)
    p.add(1)
    batches = [[rng.integers(0, 32000, size=16 * 8192, dtype=np.uint32) for _ in range(80)] for _ in range(3)]
    _run_prompts(p, batches, dt=10**7, state_every=1)


def test_shared_prefix_ending_inside_a_group():
    """Hundreds of prompts share a 35-block prefix (it ends 3 blocks into an
    8-block group) and diverge after it: their diverging blocks share that
    group's anchor and so its home bucket, which overflows into the
    key-hashed buckets.  A small index makes the overflow heavy."""
    rng = np.random.default_rng(23)
    w = _mk(n_instances=2, vnodes=16, capacity=2000, batch=200)
    p = Pair(w, max_instances=3, max_touch=8192)
    p.add(0)
    p.add(1)
    prefix = rng.integers(0, 32000, size=16 * 35, dtype=np.uint32)
    batches = []
    for _ in range(6):
        prompts = []
        for L in rng.integers(1, 21, size=200):
            prompts.append(np.concatenate([prefix, rng.integers(0, 32000, size=16 * int(L), dtype=np.uint32)]))
        batches.append(prompts)
    _run_prompts(p, batches, state_every=2)
