"""Request-sharded routing over several ranks (torch.distributed).

Each rank keeps a replica of the scheduler state (same config and seed, same
instance adds and removes, same batches).  For a batch, rank k hashes, looks
up and probes only its contiguous slice of the requests (Sec. 3.2 and
App. A.3.2 for those steps), the ranks all-gather the slices' results (per
request a few words, plus the prefix values of its blocks that the commit
needs), and every rank then runs the choice, queues, metrics and commit on
the whole batch, in arrival order, so the replicas stay identical.  The only
collective is that one all-gather per batch (NCCL between GPUs, gloo on
CPU); nothing reads another GPU's memory.

The per-rank work goes through a backend with four calls:
    begin(batch, r0, r1)      route requests r0 .. r1-1 of the batch
    export(r0, r1)            this rank's results, a 1-D uint8 tensor
    import_(r0, r1, payload)  another rank's results
    finish(batch)             the rest of the step on the whole batch
DeviceShard is the product backend (libdualmap's dm_route_shard_* calls on
a Scheduler's handle); any object with the same calls can stand in.
"""

import torch
import torch.distributed as dist

from . import dualmap as D


def shard_ranges(n, world):
    """Contiguous request ranges [r0, r1) of a batch of n, one per rank, as
    equal as integer division makes them."""
    return [(n * k // world, n * (k + 1) // world) for k in range(world)]


def all_gather_bytes(payload, group=None):
    """All-gather of 1-D uint8 tensors whose lengths differ between ranks:
    the lengths first, then the payloads padded to the longest."""
    world = dist.get_world_size(group)
    size = torch.tensor([payload.numel()], dtype=torch.int64, device=payload.device)
    sizes = [torch.zeros_like(size) for _ in range(world)]
    dist.all_gather(sizes, size, group=group)
    lens = [int(x.item()) for x in sizes]
    buf = torch.zeros(max(max(lens), 1), dtype=torch.uint8, device=payload.device)
    buf[:payload.numel()] = payload
    outs = [torch.empty_like(buf) for _ in range(world)]
    dist.all_gather(outs, buf, group=group)
    return [o[:m] for o, m in zip(outs, lens)]


class ShardedRouter:
    """Routes each batch with the requests split over the ranks of `group`."""

    def __init__(self, backend, group=None):
        self.backend = backend
        self.group = group

    def route(self, batch):
        rank = dist.get_rank(self.group)
        world = dist.get_world_size(self.group)
        ranges = shard_ranges(batch["n"], world)
        r0, r1 = ranges[rank]
        self.backend.begin(batch, r0, r1)
        parts = all_gather_bytes(self.backend.export(r0, r1), self.group)
        for k, (a, b) in enumerate(ranges):
            if k != rank and b > a:
                self.backend.import_(a, b, parts[k])
        return self.backend.finish(batch)


class DeviceShard:
    """Backend on a Scheduler (scheduler.py) and its device: a batch is a
    dict of device tensors tokens, offsets, lengths and the ints n,
    total_tokens, t (the arguments of Scheduler.route)."""

    def __init__(self, sched):
        self.g = sched
        self.b = None

    def _check(self, rc, what):
        if rc:
            raise D.DualMapError(rc, what)

    def begin(self, batch, r0, r1):
        self.b = D.make_batch(batch["tokens"], batch["offsets"], batch["lengths"], batch["n"],
                              batch["total_tokens"], batch["t"])
        self._batch = batch   # keeps the tensors alive while the handle uses them
        self._check(D.dm_route_shard_begin(self.g.h, self.b, r0, r1), "dm_route_shard_begin")

    def export(self, r0, r1):
        dev = self.g.device
        B = self.g.cfg.block_tokens
        if r1 <= r0:
            return torch.zeros(0, dtype=torch.uint8, device=dev)
        # an upper bound of the payload: every token of the batch in full blocks
        # of this range, every segment (64 blocks, plus a ragged one per request)
        nblk = int(self._batch["total_tokens"]) // B
        nseg = nblk // 64 + (r1 - r0)
        cap = 8 * (nblk + nseg) + 4 * (nseg + 5 * (r1 - r0))
        buf = torch.empty(cap, dtype=torch.uint8, device=dev)
        nbytes = torch.zeros(1, dtype=torch.int64, device=dev)
        self._check(D.dm_shard_export(self.g.h, r0, r1, buf, cap, nbytes), "dm_shard_export")
        return buf[:int(nbytes.item())]

    def import_(self, r0, r1, payload):
        self._check(D.dm_shard_import(self.g.h, r0, r1, payload, payload.numel()), "dm_shard_import")

    def finish(self, batch):
        self._check(D.dm_route_shard_finish(self.g.h, self.b, self.g.out_struct), "dm_route_shard_finish")
        self._batch = None
        return self.g.results(batch["n"])
