"""Convenience wrapper of one dm_handle with torch-owned device buffers.

Only marshalling: it allocates output tensors on the device, builds the
C structs, calls the C ABI and raises on error statuses.
"""

import ctypes as C

import torch

from . import dualmap as D

OUT_FIELDS = [("cand1", torch.int32), ("cand2", torch.int32), ("hit1", torch.int32), ("hit2", torch.int32),
              ("ttft1", torch.int64), ("ttft2", torch.int64), ("chosen", torch.int32), ("switched", torch.uint8)]


class Scheduler:
    def __init__(self, *, block_tokens=16, route_prefix_blocks=16, vnodes=64, max_instances=16,
                 capacity=65536, slo_us=2_000_000, cost_us=1, hot_num=3, hot_den=2, max_batch=4096,
                 max_batch_tokens=1 << 24, max_touch_per_instance=0, max_queue=0, index_slots_log2=0, seed=0,
                 choice_rule=0, adapt_step_blocks=0, adapt_max_blocks=0, adapt_window=1, rebalance_flags=0,
                 rebuild_pool=0, test_loop_limit=0, candidates=0, rebalance_key_blocks=0, stream=None,
                 device="cuda"):
        self.device = torch.device(device)
        self.stream = stream if stream is not None else torch.cuda.current_stream(self.device)
        self.cfg = D.dm_config(block_tokens=block_tokens, route_prefix_blocks=route_prefix_blocks,
                               vnodes_per_instance=vnodes, max_instances=max_instances,
                               cache_capacity_blocks=capacity, slo_us=slo_us, cost_us_per_token=cost_us,
                               hot_num=hot_num, hot_den=hot_den, max_batch=max_batch,
                               max_batch_tokens=max_batch_tokens, max_touch_per_instance=max_touch_per_instance,
                               max_queue=max_queue, index_slots_log2=index_slots_log2, choice_rule=choice_rule,
                               adapt_step_blocks=adapt_step_blocks, adapt_max_blocks=adapt_max_blocks,
                               adapt_window=adapt_window, rebalance_flags=rebalance_flags, rebuild_pool=rebuild_pool,
                               test_loop_limit=test_loop_limit, candidates=candidates,
                               rebalance_key_blocks=rebalance_key_blocks, seed=seed,
                               stream=C.c_void_p(self.stream.cuda_stream))
        self.h = D.dm_create(self.cfg)
        self.M = max_instances
        self.max_batch = max_batch
        self.out = {k: torch.zeros(max_batch, dtype=t, device=self.device) for k, t in OUT_FIELDS}
        self.out_struct = D.make_out(*[self.out[k] for k, _ in OUT_FIELDS])
        self.mig = torch.zeros(1 << 16, 2, dtype=torch.int64, device=self.device)   # 16-byte records
        self.mig_n = torch.zeros(1, dtype=torch.int32, device=self.device)

    def close(self):
        if self.h:
            D.dm_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def add_instance(self, i):
        return D.dm_add_instance(self.h, i)

    def remove_instance(self, i):
        return D.dm_remove_instance(self.h, i)

    def route(self, tokens, offsets, lengths, n, total_tokens, t_batch, check=True):
        """Route one batch held in device tensors; returns the status."""
        b = D.make_batch(tokens, offsets, lengths, n, total_tokens, t_batch)
        rc = D.dm_route_batch(self.h, b, self.out_struct)
        if check and rc:
            raise D.DualMapError(rc, "dm_route_batch")
        return rc

    def route_d(self, tokens, offsets, lengths, n, total_tokens, t_batch, check=True):
        """Route one batch with d candidates (dm_route_batch_d); returns the
        status.  results_d(n) reads the outputs."""
        d = self.cfg.candidates or 2
        if getattr(self, "out_d", None) is None:
            self.out_d = {"cand": torch.zeros(self.max_batch * d, dtype=torch.int32, device=self.device),
                          "hit": torch.zeros(self.max_batch * d, dtype=torch.int32, device=self.device),
                          "ttft": torch.zeros(self.max_batch * d, dtype=torch.int64, device=self.device),
                          "chosen": torch.zeros(self.max_batch, dtype=torch.int32, device=self.device),
                          "switched": torch.zeros(self.max_batch, dtype=torch.uint8, device=self.device)}
            self.out_d_struct = D.dm_route_out_d(*[self.out_d[k].data_ptr() for k in
                                                   ("cand", "hit", "ttft", "chosen", "switched")])
        b = D.make_batch(tokens, offsets, lengths, n, total_tokens, t_batch)
        rc = D.dm_route_batch_d(self.h, b, self.out_d_struct)
        if check and rc:
            raise D.DualMapError(rc, "dm_route_batch_d")
        return rc

    def results_d(self, n):
        """Host copies (numpy) of the last dm_route_batch_d outputs (n x d arrays and n vectors)."""
        torch.cuda.synchronize(self.device)
        d = self.cfg.candidates or 2
        out = {k: self.out_d[k][:n * d].cpu().numpy().reshape(n, d) for k in ("cand", "hit", "ttft")}
        out.update({k: self.out_d[k][:n].cpu().numpy() for k in ("chosen", "switched")})
        return out

    def results(self, n):
        """Host copies (numpy) of the last batch's outputs."""
        torch.cuda.synchronize(self.device)
        return {k: self.out[k][:n].cpu().numpy() for k, _ in OUT_FIELDS}

    def route_blocks(self, n):
        """Hash prefix length (blocks) of each request of the last batch (numpy)."""
        k = torch.zeros(max(n, 1), dtype=torch.int32, device=self.device)
        rc = D.dm_get_route_blocks(self.h, k, n)
        if rc:
            raise D.DualMapError(rc, "dm_get_route_blocks")
        torch.cuda.synchronize(self.device)
        return k[:n].cpu().numpy().astype("uint32")

    def rebalance(self):
        rc = D.dm_rebalance_async(self.h, self.mig, self.mig.shape[0], self.mig_n)
        if rc:
            raise D.DualMapError(rc, "dm_rebalance_async")

    def migrations(self):
        torch.cuda.synchronize(self.device)
        n = int(self.mig_n.item())
        m = self.mig[:min(n, self.mig.shape[0])].cpu().numpy()
        seq = m[:, 0].astype("uint64")
        fr = (m[:, 1].astype("uint64") & 0xFFFFFFFF).astype("uint32")
        to = (m[:, 1].astype("uint64") >> 32).astype("uint32")
        return n, (seq, fr, to)

    def commit(self):
        rc = D.dm_commit_cache(self.h)
        if rc:
            raise D.DualMapError(rc, "dm_commit_cache")

    def last_error(self):
        return D.dm_last_error(self.h)

    def loads(self):
        return D.dm_get_loads(self.h, self.M)
