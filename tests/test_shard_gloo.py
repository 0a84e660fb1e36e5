"""The request-sharded split (paper_2602_06502_gb300/shard.py) on two gloo
ranks on the CPU.  Each rank's backend is the CPU oracle: or_route_part
computes its slice's keys, hash lengths, candidates and hits, the ranks
exchange them through shard.py's all-gather, and or_route_given runs the
rest of the step on the whole batch.  After every batch and commit, every
rank's decisions, loads, queues and resident keys must equal those of an
unsharded run (or_route_batch) bit for bit.  Also the oracle halves
themselves: or_route_given after or_route_part over the whole batch is
or_route_batch."""

import os
import sys

import numpy as np
import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

from oracle.oracle import Oracle, config_from_workload  # noqa: E402
from tracegen import Trace, workload  # noqa: E402

FIELDS = ("K", "cand1", "cand2", "hit1", "hit2")


class OracleShard:
    """shard.py backend on one oracle state; a batch is a dict with the host
    arrays tokens, offsets, lengths and the ints n and t."""

    def __init__(self, ora):
        self.ora = ora
        self.parts = {}

    def begin(self, batch, r0, r1):
        self.parts = {}
        rc, part = self.ora.route_part(batch["tokens"], batch["offsets"], batch["lengths"], r0, r1)
        assert rc == 0, rc
        self.parts[(r0, r1)] = part

    def export(self, r0, r1):
        import torch
        p = self.parts[(r0, r1)]
        raw = b"".join(p[f].astype(np.uint32).tobytes() for f in FIELDS) + p["keys"].astype(np.uint64).tobytes()
        return torch.frombuffer(bytearray(raw), dtype=torch.uint8) if raw else torch.zeros(0, dtype=torch.uint8)

    def import_(self, r0, r1, payload):
        raw = payload.numpy().tobytes()
        k = r1 - r0
        p = {}
        for i, f in enumerate(FIELDS):
            p[f] = np.frombuffer(raw[4 * k * i:4 * k * (i + 1)], dtype=np.uint32)
        p["keys"] = np.frombuffer(raw[4 * k * len(FIELDS):], dtype=np.uint64)
        self.parts[(r0, r1)] = p

    def finish(self, batch):
        order = sorted(self.parts)
        cat = {f: np.concatenate([self.parts[r][f] for r in order]) for f in FIELDS + ("keys",)}
        rc, out = self.ora.route_given(batch["lengths"], batch["t"], cat["K"], cat["cand1"], cat["cand2"],
                                       cat["hit1"], cat["hit2"], cat["keys"])
        assert rc == 0, rc
        out.update({f: cat[f] for f in ("cand1", "cand2", "hit1", "hit2")})
        return out


def _oracle(w):
    o = Oracle(**config_from_workload(w))
    for i in range(w["n_instances"]):
        assert o.add_instance(i) == 0
    return o


def _snapshot(o, w):
    loads = o.loads()
    queues = [o.queue(i, cap=1 << 14)[0].tolist() for i in range(w["n_instances"])]
    caches = [sorted(o.cache(i)[0].tolist()) for i in (0, 1, 2)]
    return loads.tolist(), queues, caches


def _run(w, batches, router=None, ora=None):
    """Outputs and state after each batch and commit, routed sharded (router)
    or in one piece (ora)."""
    tr = Trace(w)
    rec = []
    for b in range(batches):
        s, e, off, lens, nt = tr.batch_layout(b)
        batch = dict(tokens=tr.batch_tokens(b), offsets=off, lengths=lens, n=e - s, t=tr.batch_time(b))
        if router is not None:
            out = router.route(batch)
            o = router.backend.ora
        else:
            rc, out = ora.route_batch(batch["tokens"], off, lens, batch["t"])
            assert rc == 0
            o = ora
        assert o.commit() == 0
        rec.append(({k: np.asarray(out[k]).tolist() for k in ("cand1", "cand2", "hit1", "hit2", "ttft1", "ttft2",
                                                               "chosen", "switched")}, _snapshot(o, w)))
    return rec


def _worker(rank, world, port, w, batches, q):
    import torch.distributed as dist
    sys.path.insert(0, ROOT)
    from paper_2602_06502_gb300.shard import ShardedRouter
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        rec = _run(w, batches, router=ShardedRouter(OracleShard(_oracle(w))))
        q.put((rank, rec))
        dist.barrier()
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_equal_the_unsharded_run():
    w = workload("tiny", n_requests=6 * 256, capacity=4000)
    batches = 6
    ref = _run(w, batches, ora=_oracle(w))
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = 29700 + os.getpid() % 1000
    procs = [ctx.Process(target=_worker, args=(r, 2, port, w, batches, q)) for r in range(2)]
    for p in procs:
        p.start()
    got = dict(q.get(timeout=300) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for r in (0, 1):
        assert len(got[r]) == batches
        for b in range(batches):
            assert got[r][b][0] == ref[b][0], (r, b)      # every decision
            assert got[r][b][1] == ref[b][1], (r, b)      # loads, queues, resident keys


def test_oracle_halves_compose_to_the_whole_step():
    w = workload("tiny", n_requests=3 * 256)
    tr = Trace(w)
    a, b = _oracle(w), _oracle(w)
    for bi in range(3):
        s, e, off, lens, nt = tr.batch_layout(bi)
        tok, t = tr.batch_tokens(bi), tr.batch_time(bi)
        rc, whole = a.route_batch(tok, off, lens, t)
        assert rc == 0
        rc, part = b.route_part(tok, off, lens, 0, e - s)
        assert rc == 0
        rc, rest = b.route_given(lens, t, part["K"], part["cand1"], part["cand2"], part["hit1"], part["hit2"],
                                 part["keys"])
        assert rc == 0
        for f in ("cand1", "cand2", "hit1", "hit2"):
            assert np.array_equal(whole[f], part[f])
        for f in ("ttft1", "ttft2", "chosen", "switched"):
            assert np.array_equal(whole[f], rest[f])
        assert a.commit() == 0 and b.commit() == 0
        assert _snapshot(a, w) == _snapshot(b, w)
        assert np.array_equal(a.route_blocks(), b.route_blocks())


def test_shard_ranges_partition_the_batch():
    from paper_2602_06502_gb300.shard import shard_ranges
    for n in (0, 1, 5, 512, 4097):
        for world in (1, 2, 3, 8):
            rs = shard_ranges(n, world)
            assert rs[0][0] == 0 and rs[-1][1] == n
            assert all(a[1] == b[0] for a, b in zip(rs, rs[1:]))
            assert max(b - a for a, b in rs) - min(b - a for a, b in rs) <= 1
