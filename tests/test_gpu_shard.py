"""The request-sharded split on the GPU path (dm_route_shard_begin,
dm_shard_export / dm_shard_import, dm_route_shard_finish, driven by
shard.py's DeviceShard).  One GPU holds two or three handles that act as
the ranks: each begins the batch on its own request range, they exchange
their exported results device to device, and each finishes the batch.  The
handles run one after the other on the same stream order; no kernel waits
for another.  Every handle's outputs, loads, queues and resident keys must
equal those of an unsharded handle (itself in parity with the oracle in
test_gpu_parity.py), batch after batch, with commits, rebalancing, index
eviction and instance changes in between."""

import numpy as np
import pytest

from parity_harness import lib_ready
from tracegen import Trace, workload

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    lib_ready()


def _sched(w, mbt, max_touch):
    from paper_2602_06502_gb300.scheduler import Scheduler
    return Scheduler(block_tokens=w["block_tokens"], route_prefix_blocks=w["route_prefix_blocks"], vnodes=w["vnodes"],
                     max_instances=w["n_instances"] + 8, capacity=w["capacity"], slo_us=w["slo_us"],
                     cost_us=w["cost_us"], max_batch=w["batch"], max_batch_tokens=mbt,
                     max_touch_per_instance=max_touch, seed=w["seed"])


def _state(g, M):
    from paper_2602_06502_gb300 import dualmap as D
    W = D.dm_get_loads(g.h, M)
    qs = [[a.tolist() for a in D.dm_export_queue(g.h, i, 1 << 14)] for i in range(4)]
    cs = [sorted(zip(*[a.tolist() for a in D.dm_export_cache(g.h, i)])) for i in range(3)]
    return W.tolist(), qs, cs


def _run(w, batches, nshards, mbt, max_touch, rebalance=False, events=()):
    import torch
    from paper_2602_06502_gb300 import dualmap as D
    from paper_2602_06502_gb300.shard import DeviceShard, shard_ranges
    tr = Trace(w)
    ref = _sched(w, mbt, max_touch)
    ranks = [DeviceShard(_sched(w, mbt, max_touch)) for _ in range(nshards)]
    every = [ref] + [r.g for r in ranks]
    for i in range(w["n_instances"]):
        for g in every:
            assert g.add_instance(i) == 0
    dev = torch.device("cuda:0")
    for b in range(batches):
        for (at, op, i) in events:
            if at == b:
                for g in every:
                    assert (g.add_instance(i) if op == "add" else g.remove_instance(i)) == 0
        s, e, off, lens, nt = tr.batch_layout(b)
        tok = torch.from_numpy(tr.batch_tokens(b).view(np.int32)).to(dev)
        offd = torch.from_numpy(off.view(np.int64)).to(dev)
        lensd = torch.from_numpy(lens.view(np.int32)).to(dev)
        n, t = e - s, tr.batch_time(b)
        ref.route(tok, offd, lensd, n, nt, t)
        want = ref.results(n)
        batch = dict(tokens=tok, offsets=offd, lengths=lensd, n=n, total_tokens=nt, t=t)
        rr = shard_ranges(n, nshards)
        for k, r in enumerate(ranks):
            r.begin(batch, *rr[k])
        pay = [r.export(*rr[k]) for k, r in enumerate(ranks)]
        for k, r in enumerate(ranks):
            for j in range(nshards):
                if j != k and rr[j][1] > rr[j][0]:
                    r.import_(rr[j][0], rr[j][1], pay[j])
        for k, r in enumerate(ranks):
            got = r.finish(batch)
            for f in want:
                assert np.array_equal(got[f], want[f]), (b, k, f)
        if rebalance:
            m0 = D.dm_rebalance(ref.h, 1 << 12)
            for r in ranks:
                m = D.dm_rebalance(r.g.h, 1 << 12)
                assert m[0] == m0[0] == 0 and m[1] == m0[1]
                assert np.array_equal(m[2], m0[2]), b
        for g in every:
            assert D.dm_commit_cache(g.h) == 0
        st = _state(ref, w["n_instances"] + 8)
        for r in ranks:
            assert _state(r.g, w["n_instances"] + 8) == st, b
            assert D.dm_last_error(r.g.h) == 0
    return ranks


def test_two_shards_tiny_with_eviction_and_rebalance():
    w = workload("tiny", n_requests=2000, batch=100, capacity=700, zipf_s=1.3, rho=1.2)
    _run(w, 12, 2, 1 << 24, 2600, rebalance=True)


def test_three_shards_agent_batches():
    w = workload("agent", n_requests=3 * 4096)
    _run(w, 3, 3, 40_000_000, 1 << 20)


def test_two_shards_long_prompts_and_instance_changes():
    w = workload("longctx", n_requests=3 * 512)
    w["capacity"] = 200_000
    _run(w, 3, 2, 70_000_000, 1 << 20, events=((1, "remove", 5), (2, "add", 130)))


def test_shard_calls_check_their_order():
    import torch
    from paper_2602_06502_gb300 import dualmap as D
    from paper_2602_06502_gb300.shard import DeviceShard
    w = workload("tiny", n_requests=256)
    tr = Trace(w)
    g = _sched(w, 1 << 24, 0)
    for i in range(w["n_instances"]):
        assert g.add_instance(i) == 0
    s, e, off, lens, nt = tr.batch_layout(0)
    dev = torch.device("cuda:0")
    tok = torch.from_numpy(tr.batch_tokens(0).view(np.int32)).to(dev)
    offd = torch.from_numpy(off.view(np.int64)).to(dev)
    lensd = torch.from_numpy(lens.view(np.int32)).to(dev)
    b = D.make_batch(tok, offd, lensd, e - s, nt, tr.batch_time(0))
    assert D.dm_route_shard_finish(g.h, b, g.out_struct) == D.DM_ERR_INVALID_ARG   # nothing begun
    assert D.dm_route_shard_begin(g.h, b, 5, 3) == D.DM_ERR_INVALID_ARG          # r0 > r1
    assert D.dm_route_shard_begin(g.h, b, 0, e - s + 1) == D.DM_ERR_INVALID_ARG  # past the batch
    assert D.dm_route_shard_begin(g.h, b, 0, 100) == 0
    assert D.dm_route_batch(g.h, b, g.out_struct) == D.DM_ERR_ORDER              # a shard is open
    assert D.dm_commit_cache(g.h) == D.DM_ERR_ORDER
    assert D.dm_add_instance(g.h, 20) == D.DM_ERR_ORDER
    small = torch.zeros(64, dtype=torch.uint8, device=dev)
    nb = torch.zeros(1, dtype=torch.int64, device=dev)
    assert D.dm_shard_export(g.h, 0, 100, small, 64, nb) == 0
    assert D.dm_last_error(g.h) == D.DM_ERR_CAPACITY                              # buffer too small: sticky
    assert int(nb.item()) > 64
    g.close()
    g = _sched(w, 1 << 24, 0)
    for i in range(w["n_instances"]):
        assert g.add_instance(i) == 0
    r = DeviceShard(g)
    batch = dict(tokens=tok, offsets=offd, lengths=lensd, n=e - s, total_tokens=nt, t=tr.batch_time(0))
    r.begin(batch, 0, e - s)                                                       # one rank: the whole batch
    r.finish(batch)
    assert D.dm_commit_cache(g.h) == 0
    assert D.dm_last_error(g.h) == 0
