"""Run the same seeded trace through the CPU oracle and the CUDA library (via
its C ABI) and compare every result bit for bit."""

import numpy as np

from oracle import oracle as O

OUT_KEYS = ["cand1", "cand2", "hit1", "hit2", "ttft1", "ttft2", "chosen", "switched"]


def lib_ready():
    import __graft_entry__ as g
    g.build()


class Pair:
    """An oracle and a GPU scheduler built from the same workload dict."""

    def __init__(self, w, max_instances=None, max_batch_tokens=None, max_touch=0, max_queue=0, capacity=None,
                 index_slots_log2=0, choice_rule=0, adapt=None, rebalance_flags=0, rebuild_pool=0,
                 rebalance_key_blocks=0):
        import torch
        from paper_2602_06502_gb300.scheduler import Scheduler
        self.torch = torch
        self.w = dict(w)
        if capacity is not None:
            self.w["capacity"] = capacity
        w = self.w
        self.M = max_instances or (w["n_instances"] + 8)
        mbt = max_batch_tokens or (1 << 24)
        ad = dict(adapt_step_blocks=0, adapt_max_blocks=0, adapt_window=1) if adapt is None else dict(adapt)
        self.adaptive = bool(ad["adapt_step_blocks"])
        self.ora = O.Oracle(**O.config_from_workload(w, max_instances=self.M, max_batch_tokens=mbt),
                            choice_rule=choice_rule, rebalance_flags=rebalance_flags, **ad)
        self.gpu = Scheduler(block_tokens=w["block_tokens"], route_prefix_blocks=w["route_prefix_blocks"],
                             vnodes=w["vnodes"], max_instances=self.M, capacity=w["capacity"], slo_us=w["slo_us"],
                             cost_us=w["cost_us"], max_batch=w["batch"], max_batch_tokens=mbt,
                             max_touch_per_instance=max_touch, max_queue=max_queue,
                             index_slots_log2=index_slots_log2, seed=w["seed"], choice_rule=choice_rule,
                             rebalance_flags=rebalance_flags, rebuild_pool=rebuild_pool,
                             rebalance_key_blocks=rebalance_key_blocks, **ad)
        self.dev = torch.device("cuda:0")
        self.n_migrations = 0
        self.n_switched = 0
        self.hit_tokens = 0

    def add(self, i):
        a, b = self.ora.add_instance(i), self.gpu.add_instance(i)
        assert a == b, (i, a, b)
        return a

    def remove(self, i):
        a, b = self.ora.remove_instance(i), self.gpu.remove_instance(i)
        assert a == b, (i, a, b)
        return a

    def to_dev(self, tok, off, lens):
        t = self.torch
        tok = np.ascontiguousarray(tok, dtype=np.uint32)
        return (t.from_numpy(tok.view(np.int32) if tok.size else np.zeros(4, np.int32)).to(self.dev),
                t.from_numpy(np.ascontiguousarray(off, dtype=np.uint64).view(np.int64)).to(self.dev),
                t.from_numpy(np.ascontiguousarray(lens, dtype=np.uint32).view(np.int32)).to(self.dev))

    def route(self, tok, off, lens, t_batch, tag=""):
        n = len(lens)
        rc, want = self.ora.route_batch(tok, off, lens, t_batch)
        assert rc == 0, rc
        dt, do, dl = self.to_dev(tok, off, lens)
        self.gpu.route(dt, do, dl, n, max(len(tok), 4), t_batch)
        got = self.gpu.results(n)
        assert self.gpu.last_error() == 0, tag
        for k in OUT_KEYS:
            g = got[k].astype(want[k].dtype)
            if not np.array_equal(g, want[k]):
                bad = np.nonzero(g != want[k])[0]
                raise AssertionError(f"{tag}: {k} differs at {bad[:8].tolist()} "
                                     f"(gpu {g[bad[:4]].tolist()} vs oracle {want[k][bad[:4]].tolist()})")
        gk, ok = self.gpu.route_blocks(n), self.ora.route_blocks()
        if not np.array_equal(gk, ok):
            bad = np.nonzero(gk != ok)[0]
            raise AssertionError(f"{tag}: route blocks differ at {bad[:8].tolist()} "
                                 f"(gpu {gk[bad[:4]].tolist()} vs oracle {ok[bad[:4]].tolist()})")
        if self.adaptive:
            from paper_2602_06502_gb300 import dualmap as D
            assert np.array_equal(D.dm_export_prefix_tree(self.gpu.h), self.ora.prefix_tree()), f"{tag}: tree"
        self.n_switched += int(want["switched"].sum())
        self.hit_tokens += int(np.where(want["chosen"] == want["cand1"], want["hit1"], want["hit2"]).sum())
        return want

    def rebalance(self, tag=""):
        rc, n, (seq, fr, to) = self.ora.rebalance()
        assert rc == 0
        self.gpu.rebalance()
        gn, (gseq, gfr, gto) = self.gpu.migrations()
        assert gn == n, f"{tag}: {gn} vs {n} migrations (GPU status {self.gpu.last_error()}; oracle {seq.tolist()})"
        assert np.array_equal(gseq, seq) and np.array_equal(gfr, fr) and np.array_equal(gto, to), tag
        self.n_migrations += n
        return n

    def commit(self):
        assert self.ora.commit() == 0
        self.gpu.commit()

    def check_loads(self, tag=""):
        assert self.gpu.last_error() == 0, tag
        assert np.array_equal(self.gpu.loads(), self.ora.loads()), tag

    def check_metrics(self, tag=""):
        """Serving metrics: every counter, the TTFT histogram and the CV
        samples (floating point, bit for bit)."""
        from paper_2602_06502_gb300 import dualmap as D
        gm, gh = D.dm_get_metrics(self.gpu.h)
        om, oh = self.ora.metrics()
        assert np.array_equal(gh, oh), f"{tag}: TTFT histogram"
        for k in O.METRIC_KEYS:
            assert gm[k] == om[k], f"{tag}: {k} gpu {gm[k]} vs oracle {om[k]}"
        for k in ("cv_sum", "cv_last"):
            assert gm[k] == om[k], f"{tag}: {k} gpu {gm[k]!r} vs oracle {om[k]!r}"
        return om

    def check_state(self, ids=None, tag=""):
        """Loads, queues (seq, work, remaining), resident (key, stamp) sets, clock."""
        from paper_2602_06502_gb300 import dualmap as D
        self.check_loads(tag)
        assert D.dm_get_clock(self.gpu.h) == self.ora.clock(), tag
        for i in (range(self.M) if ids is None else ids):
            qs = self.ora.queue(i)
            gs = D.dm_export_queue(self.gpu.h, i)
            for a, b in zip(qs, gs):
                assert np.array_equal(a, b), f"{tag}: queue {i}"
            ok, os_ = self.ora.cache(i)
            gk, gs_ = D.dm_export_cache(self.gpu.h, i)
            o = np.lexsort((ok, os_))
            g = np.lexsort((gk, gs_))
            assert np.array_equal(ok[o], gk[g]) and np.array_equal(os_[o], gs_[g]), f"{tag}: cache {i}"


def run_trace(pair, tr, batches=None, rebalance=None, state_every=0, check_state_end=True):
    """Replay trace batches (with its add/remove events) on both sides."""
    w = tr.cfg
    if rebalance is None:
        rebalance = w.get("rebalance", False)
    for i in range(w["n_instances"]):
        assert pair.add(i) == 0
    events = {}
    for b, kind, i in tr.events:
        events.setdefault(b, []).append((kind, i))
    nb = len(tr.batches) if batches is None else min(batches, len(tr.batches))
    for b in range(nb):
        for kind, i in events.get(b, []):
            assert (pair.add(i) if kind == "add" else pair.remove(i)) == 0
        s, e, off, lens, ntok = tr.batch_layout(b)
        pair.route(tr.batch_tokens(b), off, lens, tr.batch_time(b), tag=f"batch {b}")
        if rebalance:
            pair.rebalance(tag=f"batch {b}")
        pair.commit()
        pair.check_loads(tag=f"batch {b}")
        if state_every and (b + 1) % state_every == 0:
            pair.check_state(tag=f"batch {b}")
            pair.check_metrics(tag=f"batch {b}")
    if check_state_end:
        pair.check_state(tag="end")
    return pair.check_metrics(tag="end")
