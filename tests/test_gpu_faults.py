"""Failure handling on the device and on allocation, made to happen in safe
ways: a bounded device loop made to give up (a test-only cap on the index's
bucket walks and touch retries) must end as a sticky DM_ERR_TIMEOUT that
state-changing calls return and read-only calls survive; an allocation made
to fail (the dm_test_fail_alloc hook, no real exhaustion) must end as
DM_ERR_OOM with no handle state left behind.  No kernel is made to fault,
trap or hang."""

import ctypes as C

import numpy as np
import pytest

from parity_harness import lib_ready

pytestmark = pytest.mark.gpu


def _one_block_batch(torch, n, B, seed):
    rng = np.random.default_rng(seed)
    tok = rng.integers(0, 1 << 32, size=n * B + 4, dtype=np.uint64).astype(np.uint32)
    off = (np.arange(n, dtype=np.uint64) * B)
    lens = np.full(n, B, np.uint32)
    dev = torch.device("cuda:0")
    return (torch.from_numpy(tok.view(np.int32)).to(dev), torch.from_numpy(off.view(np.int64)).to(dev),
            torch.from_numpy(lens.view(np.int32)).to(dev), n * B)


def _tiny(limit):
    from paper_2602_06502_gb300.scheduler import Scheduler
    # 8 buckets of 8 slots per index (2 x (C + T) = 64): 24 one-block prompts
    # over 2 instances put at least two keys into one bucket of one index
    g = Scheduler(block_tokens=16, route_prefix_blocks=1, vnodes=4, max_instances=4, capacity=8,
                  max_touch_per_instance=24, max_batch=32, max_batch_tokens=1 << 12, max_queue=256, seed=3,
                  test_loop_limit=limit)
    for i in range(2):
        assert g.add_instance(i) == 0
    return g


def test_a_bounded_loop_that_gives_up_is_a_sticky_timeout():
    lib_ready()
    import torch
    from paper_2602_06502_gb300 import dualmap as D
    tok, off, lens, ntok = _one_block_batch(torch, 24, 16, 7)
    ok = _tiny(0)                        # control: the default bounds never give up here
    ok.route(tok, off, lens, 24, ntok, 100)
    ok.commit()
    assert ok.last_error() == D.DM_OK
    ok.close()
    g = _tiny(1)                         # one step per walk: a displaced touch gives up
    g.route(tok, off, lens, 24, ntok, 100)
    g.commit()
    assert g.last_error() == D.DM_ERR_TIMEOUT
    assert g.last_error() == D.DM_ERR_TIMEOUT                   # sticky
    b = D.make_batch(tok, off, lens, 24, ntok, 200)
    assert D.dm_route_batch(g.h, b, g.out_struct) == D.DM_ERR_TIMEOUT
    assert D.dm_commit_cache(g.h) == D.DM_ERR_TIMEOUT
    assert D.dm_add_instance(g.h, 3) == D.DM_ERR_TIMEOUT
    # read-only calls still answer
    assert len(D.dm_get_loads(g.h, 4)) == 4
    clk = C.c_uint64()
    assert D.lib().dm_get_clock(g.h, C.byref(clk)) == D.DM_OK
    n = C.c_uint64()
    assert D.lib().dm_export_queue(g.h, 0, None, None, None, 0, C.byref(n)) == D.DM_OK
    g.close()


def test_allocation_failures_return_oom_and_leave_nothing_behind():
    lib_ready()
    import torch
    from paper_2602_06502_gb300 import dualmap as D
    cfg = D.dm_config(block_tokens=16, route_prefix_blocks=4, vnodes_per_instance=8, max_instances=8,
                      cache_capacity_blocks=1024, slo_us=1000, cost_us_per_token=1, hot_num=3, hot_den=2,
                      max_batch=64, max_batch_tokens=1 << 16, seed=5,
                      stream=C.c_void_p(torch.cuda.current_stream().cuda_stream))
    torch.cuda.synchronize()
    free0 = torch.cuda.mem_get_info()[0]
    h = C.c_void_p()
    try:
        # dm_create fails at its first, a middle and a late allocation
        for k in (0, 7, 40):
            D.lib().dm_test_fail_alloc(k)
            assert D.lib().dm_create(C.byref(cfg), C.byref(h)) == D.DM_ERR_OOM, k
            assert not h.value
        D.lib().dm_test_fail_alloc(-1)
        torch.cuda.synchronize()
        assert abs(torch.cuda.mem_get_info()[0] - free0) < (64 << 20)   # everything was freed
        # dm_add_instance: the first add of an id allocates its index
        assert D.lib().dm_create(C.byref(cfg), C.byref(h)) == D.DM_OK
        assert D.lib().dm_add_instance(h, 0) == D.DM_OK
        D.lib().dm_test_fail_alloc(0)
        assert D.lib().dm_add_instance(h, 1) == D.DM_ERR_OOM
        D.lib().dm_test_fail_alloc(-1)
        # nothing of id 1 is live: it can be added afterwards, and routing works
        assert D.lib().dm_add_instance(h, 1) == D.DM_OK
        tok, off, lens, ntok = _one_block_batch(torch, 8, 16, 9)
        out = {k: torch.zeros(64, dtype=t, device="cuda") for k, t in
               [("cand1", torch.int32), ("cand2", torch.int32), ("hit1", torch.int32), ("hit2", torch.int32),
                ("ttft1", torch.int64), ("ttft2", torch.int64), ("chosen", torch.int32),
                ("switched", torch.uint8)]}
        o = D.make_out(*[out[k] for k in ("cand1", "cand2", "hit1", "hit2", "ttft1", "ttft2", "chosen",
                                          "switched")])
        assert D.dm_route_batch(h, D.make_batch(tok, off, lens, 8, ntok, 10), o) == D.DM_OK
        assert D.lib().dm_last_error(h) == D.DM_OK
        assert set(out["chosen"][:8].cpu().tolist()) <= {0, 1}
    finally:
        D.lib().dm_test_fail_alloc(-1)
        if h.value:
            D.lib().dm_destroy(h)
