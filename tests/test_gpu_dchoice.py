"""Routing with d candidates (App. A.8) on the GPU, bit for bit against the
oracle: every candidate, hit length, TTFT estimate, choice and switch flag
per request; loads after every batch; queues, resident sets, clock and
metrics at the end; the d rings through adds and removes; d = 2 through the
d-way kernels equal to DualMap's routing; and the argument checks of a
handle made for d candidates."""

import ctypes as C

import numpy as np
import pytest

from oracle import oracle as O
from parity_harness import lib_ready
from tracegen import Trace, workload

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    lib_ready()


def _pair(w, d, M, mbt, **kw):
    from paper_2602_06502_gb300.scheduler import Scheduler
    ora = O.Oracle(**O.config_from_workload(w, max_instances=M, max_batch_tokens=mbt,
                                            candidates=max(d, 2) if d != 2 else 2))
    gpu = Scheduler(block_tokens=w["block_tokens"], route_prefix_blocks=w["route_prefix_blocks"], vnodes=w["vnodes"],
                    max_instances=M, capacity=w["capacity"], slo_us=w["slo_us"], cost_us=w["cost_us"],
                    max_batch=w["batch"], max_batch_tokens=mbt, seed=w["seed"],
                    candidates=kw.get("gpu_candidates", d), max_touch_per_instance=kw.get("max_touch", 0))
    return ora, gpu


def _replay(tr, d, M=None, mbt=1 << 24, events=True, **kw):
    import torch
    from paper_2602_06502_gb300 import dualmap as D
    w = tr.cfg
    M = M or w["n_instances"] + 8
    ora, gpu = _pair(w, d, M, mbt, **kw)
    for i in range(w["n_instances"]):
        assert ora.add_instance(i) == 0 and gpu.add_instance(i) == 0
    ev = {}
    for b, kind, i in (tr.events if events else []):
        ev.setdefault(b, []).append((kind, i))
    dev = torch.device("cuda:0")
    switched = 0
    for b in range(len(tr.batches)):
        for kind, i in ev.get(b, []):
            a = ora.add_instance(i) if kind == "add" else ora.remove_instance(i)
            g = gpu.add_instance(i) if kind == "add" else gpu.remove_instance(i)
            assert a == g == 0
        s, e, off, lens, ntok = tr.batch_layout(b)
        tok = tr.batch_tokens(b)
        rc, want = ora.route_batch_d(d, tok, off, lens, tr.batch_time(b))
        assert rc == 0
        gpu.route_d(torch.from_numpy(tok.view(np.int32)).to(dev), torch.from_numpy(off.view(np.int64)).to(dev),
                    torch.from_numpy(lens.view(np.int32)).to(dev), e - s, ntok, tr.batch_time(b))
        got = gpu.results_d(e - s)
        assert gpu.last_error() == 0
        for k in ("cand", "hit", "ttft", "chosen", "switched"):
            g = got[k].astype(want[k].dtype)
            if not np.array_equal(g, want[k]):
                bad = np.argwhere(g != want[k])[:4].tolist()
                raise AssertionError(f"batch {b}: {k} differs at {bad}")
        switched += int(want["switched"].sum())
        assert ora.commit() == 0
        gpu.commit()
        assert np.array_equal(gpu.loads(), ora.loads()), f"batch {b}: loads"
    # end state: queues, resident sets, clock, metrics
    assert D.dm_get_clock(gpu.h) == ora.clock()
    for i in range(M):
        for a, g in zip(ora.queue(i), D.dm_export_queue(gpu.h, i)):
            assert np.array_equal(a, g), f"queue {i}"
        ok, os_ = ora.cache(i)
        gk, gs = D.dm_export_cache(gpu.h, i)
        o, q = np.lexsort((ok, os_)), np.lexsort((gk, gs))
        assert np.array_equal(ok[o], gk[q]) and np.array_equal(os_[o], gs[q]), f"cache {i}"
    gm, gh = D.dm_get_metrics(gpu.h)
    om, oh = ora.metrics()
    assert np.array_equal(gh, oh)
    for k in O.METRIC_KEYS:
        assert gm[k] == om[k], k
    assert gm["cv_sum"] == om["cv_sum"]
    return ora, gpu, switched


@pytest.mark.parametrize("d", [1, 3, 4])
def test_d_candidates_tiny(d):
    tr = Trace(workload("tiny", n_requests=1000, batch=200, zipf_s=1.2, rho=1.3, slo_us=40_000))
    _, gpu, sw = _replay(tr, d)
    if d > 1:
        assert sw > 0
    gpu.close()


@pytest.mark.parametrize("d", [3, 8])
def test_d_candidates_agent_batches(d):
    tr = Trace(workload("agent", n_requests=2 * 4096))
    _, gpu, _ = _replay(tr, d, mbt=40_000_000, max_touch=1 << 20)
    gpu.close()


def test_d_rings_through_adds_and_removes():
    from paper_2602_06502_gb300 import dualmap as D
    w = workload("scaling", n_requests=3 * 4096, scale_every=4096, n_instances=16, vnodes=64, capacity=20_000)
    tr = Trace(w)
    assert len(tr.events) >= 2
    ora, gpu, _ = _replay(tr, 4, M=w["n_instances"] + 4, mbt=40_000_000, max_touch=1 << 20)
    for f in range(4):
        vp, ow, _ = ora.ring(f)
        gv, go = D.dm_export_ring(gpu.h, f, 1 << 20)
        assert np.array_equal(vp, gv) and np.array_equal(ow, go), f
    gpu.close()


def test_two_candidates_through_the_d_way_kernels_are_dualmap():
    """A DualMap handle routed through dm_route_batch_d (d = 2) gives the
    oracle's DualMap decisions."""
    tr = Trace(workload("tiny", n_requests=800, batch=200, zipf_s=1.2, rho=1.3, slo_us=40_000))
    _, gpu, sw = _replay(tr, 2, gpu_candidates=0)
    assert sw > 0
    gpu.close()


def test_d_candidate_handle_argument_checks():
    import torch
    from paper_2602_06502_gb300 import dualmap as D
    from paper_2602_06502_gb300.scheduler import Scheduler
    g = Scheduler(block_tokens=16, route_prefix_blocks=4, vnodes=8, max_instances=8, capacity=64, max_batch=16,
                  max_batch_tokens=1 << 12, seed=2, candidates=5)
    for i in range(4):
        assert g.add_instance(i) == 0
    tok = torch.zeros(64 + 4, dtype=torch.int32, device="cuda")
    off = torch.zeros(1, dtype=torch.int64, device="cuda")
    ln = torch.full((1,), 64, dtype=torch.int32, device="cuda")
    b = D.make_batch(tok, off, ln, 1, 64, 10)
    assert D.dm_route_batch(g.h, b, g.out_struct) == D.DM_ERR_INVALID_ARG     # two-candidate entry point
    assert g.route_d(tok, off, ln, 1, 64, 10, check=False) == D.DM_ERR_NO_INSTANCES   # 4 live < 5
    assert g.add_instance(4) == 0
    assert g.route_d(tok, off, ln, 1, 64, 10, check=False) == D.DM_OK
    n = C.c_uint32()
    mig = (D.dm_migration * 4)()
    assert D.lib().dm_rebalance(g.h, mig, 4, C.byref(n)) == D.DM_ERR_INVALID_ARG
    assert g.last_error() == D.DM_OK
    g.close()
