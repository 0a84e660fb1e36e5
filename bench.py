"""Benchmark of the DualMap batched routing path on GB300.

One step = one batch through the whole path: queue drain, prompt hashing,
dual-ring lookup + cache probes, SLO-aware choice, (rebalance when the
workload has it) and the LRU cache commit.  Default workload: the
long-context stress shape (128 instances, 512 prompts of 32,768-131,072
uint32 tokens per batch, 64 shared 16k-token prefixes, Zipf 0.8), inputs
resident in HBM (each batch ~168 MB, larger than L2).

Prints one JSON line: routed requests/s (value), prompt GB/s hashed+probed
(hashing, ring lookup and probes are one kernel, event-timed in the timed
region) with its HBM roofline, the end-to-end number through the
host-buffer entry point, the CPU oracle baseline and the SM clocks seen.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl dualmap|reference]
  torchrun --nproc-per-node N bench.py --gpus N ...   (N independent replicas)
"""

import argparse
import hashlib
import json
import os
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "routed req/s & prompt GB/s hashed+probed on 1 GB300; % HBM roofline"
HASH_SRC = os.path.join(ROOT, "paper_2602_06502_gb300", "csrc", "dm_hash.cu")
TRAFFIC_FILE = os.path.join(ROOT, "profiles", "hash_longctx_traffic.json")


def longctx_handle_kwargs(w):
    """Handle sizes used for the long-context workload (bench and its parity test)."""
    return dict(max_instances=w["n_instances"] + 8, max_batch=w["batch"],
                max_batch_tokens=w["batch"] * w["len_hi"] + 4 * w["batch"],
                max_touch_per_instance=1 << 20, index_slots_log2=25, rebuild_pool=16)


# Opening batches after which the trace's busiest instances evict in every
# batch (long context: 42 of its 128 instances are at capacity after 56
# batches, by the oracle), routed untimed before a short run's warm-up.
STEADY_PREFILL = {"longctx": 56}


def handle_kwargs(w, max_id):
    if w["name"] == "longctx":
        return longctx_handle_kwargs(w)
    mb = w["batch"] * (w.get("len_hi") or w.get("max_prompt") or (w.get("prefix_hi", 0) + w.get("uniq_hi", 0)))
    # blocks one commit may touch on one instance: the busiest pair of a batch
    # takes well under half of it in every workload here
    touch = min(mb // w["block_tokens"], 1 << 21 if w["n_instances"] <= 64 else 1 << 19)
    return dict(max_instances=max_id + 9, max_batch=w["batch"], max_batch_tokens=mb + 4 * w["batch"],
                max_touch_per_instance=touch)


def describe_lengths(w):
    if "len_lo" in w:
        return f"{w['len_lo']}-{w['len_hi']}"
    if w["kind"] == "template":
        return f"{w['prefix_lo'] + w['uniq_lo']}-{w['prefix_hi'] + w['uniq_hi']}"
    return f"{w['chunk_lo']}-{w['max_prompt']} (multi-turn)"


def peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


def file_sha(p):
    with open(p, "rb") as f:
        return hashlib.sha256(f.read()).hexdigest()


def traffic_per_launch(token_bytes):
    """DRAM bytes (read + write) per hashing launch of `token_bytes` of
    prompts, scaled from the committed ncu capture of one full-size batch
    (traffic grows in proportion to the tokens hashed); None when the kernel
    source changed since the capture was taken."""
    try:
        with open(TRAFFIC_FILE) as f:
            t = json.load(f)
        if t.get("dm_hash_sha256") != file_sha(HASH_SRC):
            return None
        return float(t["dram_bytes_per_launch"]) * token_bytes / float(t["batch_token_bytes"])
    except Exception:
        return None


class ClockSampler:
    """nvidia-smi clocks / throttle reasons sampled in the background."""
    Q = ("timestamp,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, dev_index):
        self.rows = []
        self.proc = None
        try:
            self.proc = subprocess.Popen(["nvidia-smi", f"--query-gpu={self.Q}", "--format=csv,noheader,nounits",
                                          "-i", str(dev_index), "-lms", "50"], stdout=subprocess.PIPE,
                                         stderr=subprocess.DEVNULL, text=True)
            self.th = threading.Thread(target=self._read, daemon=True)
            self.th.start()
        except Exception:
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            parts = [x.strip() for x in line.split(",")]
            if len(parts) >= 9:
                self.rows.append((time.time(), parts))

    def stop(self):
        if self.proc:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self, t0, t1):
        inside = [p for (t, p) in self.rows if t0 <= t <= t1]
        window = "timed region"
        if not inside:
            inside = [p for (t, p) in self.rows if t0 - 1.0 <= t <= t1 + 1.0]
            window = "timed region +-1 s (region shorter than the sampling interval)"
        if not inside:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0, "window": "none"}
        sm = [float(p[1]) for p in inside if p[1].replace(".", "").isdigit()]
        mx = [float(p[2]) for p in inside if p[2].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[k] for p in inside for k in range(4) if p[5 + k].lower() == "active"})
        return {"sm_mhz": float(np.median(sm)) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": reasons, "samples": len(inside), "window": window}


def max_over_ranks(x, device="cpu"):
    """Largest value of x over the ranks of the default process group (x
    itself when not distributed): step time is the slowest replica's."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return float(x)
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(requests_per_rank, ms_max, world):
    """Whole-job routed requests/s: every replica routes the same number of
    requests, the job takes as long as its slowest replica."""
    return world * requests_per_rank / (ms_max / 1e3)


def dist_setup():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def cpu_oracle_run(tr, w, warm, timed, get_tokens, max_id, keep=None, extra=None):
    """Time the CPU oracle (as it stands, one thread) over the `timed` steps,
    after routing the `warm` steps untimed on the same state.  A step is a
    batch index, or (batch, cycle) for a pass longer than the trace, which
    replays it shifted by the trace's span in time (its instance events only
    in cycle 0).  keep: a dict that receives each batch's routing outputs
    (for the comparison with the GPU's)."""
    from oracle import oracle as O
    ora = O.Oracle(**O.config_from_workload(w, max_instances=max_id + 9, max_batch_tokens=1 << 40, **(extra or {})))
    for i in range(w["n_instances"]):
        ora.add_instance(i)
    events = {}
    for b, kind, i in tr.events:
        events.setdefault(b, []).append((kind, i))
    span = int(tr.arrival_us[-1]) + 1
    spent = 0.0
    nreq = 0
    for k, step in enumerate(list(warm) + list(timed)):
        b, cyc = step if isinstance(step, tuple) else (step, 0)
        s, e, off, lens, ntok = tr.batch_layout(b)
        tok = get_tokens(b)
        t0 = time.perf_counter()
        for kind, i in (events.get(b, []) if cyc == 0 else []):
            (ora.add_instance if kind == "add" else ora.remove_instance)(i)
        rc, out = ora.route_batch(tok, off, lens, tr.batch_time(b) + cyc * span)
        assert rc == 0
        if keep is not None:
            keep[b] = out
        if w.get("rebalance"):
            ora.rebalance()
        ora.commit()
        if k >= len(warm):
            spent += time.perf_counter() - t0
            nreq += e - s
    return nreq, spent


def run_reference(args, world, rank):
    """--impl reference: the CPU oracle timed on the host cores."""
    from tracegen import Trace, workload
    if rank != 0:
        return
    w = workload(args.workload)
    tr = Trace(w)
    nb = len(tr.batches)
    # exactly W warm-up and K timed steps of whole batches, in trace order as
    # the GPU arm runs them (cyclically past the trace's end); on the
    # long-context workload a batch takes the oracle about half a second
    # (after the same untimed cache prefill as the GPU arm's)
    P = args.prefill if args.prefill >= 0 else max(0, min(STEADY_PREFILL.get(w["name"], 0),
                                                          nb - args.warmup - args.steps))
    order = [(j % nb, j // nb) for j in range(P + args.warmup + args.steps)]
    warm, timed = order[:P + args.warmup], order[P + args.warmup:]
    k = len(timed)
    nreq, spent = cpu_oracle_run(tr, w, warm, timed, tr.batch_tokens, tr.max_instance_id())
    val = nreq / spent if spent > 0 else 0.0
    line = {"impl": "reference", "metric": METRIC, "value": val, "unit": "req/s", "n_gpus": args.gpus,
            "steps": k, "warmup": len(warm) - P, "ms_per_step": 1e3 * spent / max(k, 1), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "u32/u64 integer", "data": "synthetic",
            "config": {"workload": f"{w['name']}: {w['n_instances']} instances, batch {w['batch']}",
                       "cache_prefill_batches": P,
                       "note": "reference arm = the plain-C CPU oracle, one host thread"},
            "cpu_baseline": {"value": val, "unit": "req/s", "cores": 1, "kind": "oracle",
                             "sample": f"{k} timed batches of {w['batch']} requests after {len(warm)} untimed ones "
                                       f"({P} of them the cache prefill), in trace order"},
            "e2e": {"value": val, "unit": "req/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=120)
    ap.add_argument("--warmup", type=int, default=8)
    ap.add_argument("--impl", default="dualmap", choices=["dualmap", "reference"])
    ap.add_argument("--workload", default="longctx")
    ap.add_argument("--e2e-steps", type=int, default=24)
    ap.add_argument("--cpu-batches", type=int, default=6)
    ap.add_argument("--prefill", type=int, default=-1,
                    help="batches routed untimed before the warm-up (default: the workload's own, if it fits)")
    ap.add_argument("--no-cpu", action="store_true")
    ap.add_argument("--set", action="append", default=[], metavar="KEY=VALUE",
                    help="override a workload field (small cases for profiling)")
    ap.add_argument("--max-touch", type=int, default=0, help="override max_touch_per_instance")
    ap.add_argument("--index-slots-log2", type=int, default=0, help="override the index size (log2 slots)")
    ap.add_argument("--adapt", default="", metavar="STEP,MAX[,WINDOW]",
                    help="adaptive hash-prefix length: blocks per step, longest prefix, batches per window")
    ap.add_argument("--rule", default="dualmap",
                    help="choice rule (dualmap, pair_*, cache_affinity, least_loaded, min_ttft, preble)")
    args = ap.parse_args()
    world, rank, local = dist_setup()
    if args.impl == "reference":
        return run_reference(args, world, rank)

    import torch
    import torch.distributed as dist
    from paper_2602_06502_gb300 import dualmap as D
    from paper_2602_06502_gb300.scheduler import Scheduler, OUT_FIELDS
    import tracegen.device as TD
    from tracegen import Trace, workload

    if world > 1:
        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    w = workload(args.workload, **{k: int(v) for k, v in (x.split("=", 1) for x in args.set)})
    W, K = max(args.warmup, 3), args.steps
    tr = Trace(w)
    nb = len(tr.batches)
    kw = handle_kwargs(w, tr.max_instance_id())
    if args.max_touch:
        kw["max_touch_per_instance"] = args.max_touch
    if args.index_slots_log2:
        kw["index_slots_log2"] = args.index_slots_log2
    rule = D.RULE_NAMES.index(args.rule)
    kw["choice_rule"] = rule
    if args.adapt:
        a = [int(x) for x in args.adapt.split(",")]
        kw.update(adapt_step_blocks=a[0], adapt_max_blocks=a[1], adapt_window=a[2] if len(a) > 2 else 1)

    # cache prefill: a short run first routes the trace's opening batches
    # untimed, so that its timed steps find the instances' LRUs at capacity
    # as a long run does (never cycling past the trace's end for it)
    P = args.prefill if args.prefill >= 0 else max(0, min(STEADY_PREFILL.get(w["name"], 0), nb - W - K))
    WP = P + W   # untimed steps before the timed ones
    # all batches' tokens resident in HBM (a pass longer than the trace replays it cyclically)
    used = min(nb, WP + K)
    ntok = int(tr.req_off[tr.batches[used - 1][1]])
    tokens = torch.empty(ntok + 4, dtype=torch.int32, device=dev)
    for b0 in range(0, used, 16):
        b1 = min(used, b0 + 16)
        s0, e1 = tr.batches[b0][0], tr.batches[b1 - 1][1]
        TD.fill_range(tr, s0, e1, tokens[int(tr.req_off[s0]):int(tr.req_off[e1])])
    meta = []
    for b in range(used):
        s, e, off, lens, nt = tr.batch_layout(b)
        meta.append((s, e, torch.from_numpy(off.view(np.int64)).to(dev),
                     torch.from_numpy(lens.view(np.int32)).to(dev), nt, int(tr.req_off[s])))
    span = int(tr.arrival_us[-1]) + 1
    events = {}
    for b, kind, i in tr.events:
        events.setdefault(b, []).append((kind, i))

    def make_sched():
        g = Scheduler(block_tokens=w["block_tokens"], route_prefix_blocks=w["route_prefix_blocks"],
                      vnodes=w["vnodes"], capacity=w["capacity"], slo_us=w["slo_us"], cost_us=w["cost_us"],
                      seed=w["seed"], **kw)
        for i in range(w["n_instances"]):
            assert g.add_instance(i) == 0
        return g

    def step(g, j, host=None):
        b = j % used
        cyc = j // used
        for kind, i in (events.get(b, []) if cyc == 0 else []):
            assert (g.add_instance(i) if kind == "add" else g.remove_instance(i)) == 0
        s, e, doff, dlen, nt, t0 = meta[b]
        tb = tr.batch_time(b) + cyc * span
        if host is None:
            g.route(tokens[t0:t0 + nt + 4], doff, dlen, e - s, nt, tb)
        else:   # pinned host buffers: upload, route and readback are enqueued; uploads overlap routing
            hb = D.make_batch(host["tok"][b], host["off"][b], host["len"][b], e - s, nt, tb)
            rc = D.dm_route_batch_host_async(g.h, hb, host["out_struct"][j % 2])
            assert rc == 0, rc
        if w.get("rebalance"):
            g.rebalance()
        g.commit()
        return e - s

    # -- end-to-end through the host-buffer entry point ----------------------
    # (first, while the process's host memory is fresh: pinned upload speed on
    # this platform depends on where the pinned pages land)
    e2e = None
    if args.e2e_steps > 0:
        Ke = max(1, min(args.e2e_steps, K))
        g = make_sched()
        need = sorted({j % used for j in range(P, WP + Ke)})
        host = {"tok": {}, "off": {}, "len": {}}
        for b in need:
            s, e, doff, dlen, nt, t0 = meta[b]
            ht = torch.empty(nt + 4, dtype=torch.int32, pin_memory=True)
            ht.copy_(tokens[t0:t0 + nt + 4])
            host["tok"][b] = ht
            host["off"][b] = doff.cpu().pin_memory()
            host["len"][b] = dlen.cpu().pin_memory()
        houts = [{name: torch.zeros(w["batch"], dtype=t, pin_memory=True) for name, t in OUT_FIELDS}
                 for _ in range(2)]
        host["out_struct"] = [D.make_out(*[ho[name] for name, _ in OUT_FIELDS]) for ho in houts]
        for j in range(P):   # the prefill through the device-resident path
            step(g, j)
        for j in range(P, WP):
            step(g, j, host)
        torch.cuda.synchronize()
        h2d = d2h = 0
        t0 = time.perf_counter()
        ne = 0
        for j in range(WP, WP + Ke):
            n = step(g, j, host)
            ne += n
            b = j % used
            h2d += 4 * (meta[b][4]) + 12 * n
            d2h += 41 * n
        assert g.last_error() == 0          # synchronises the handle's stream (all copies included)
        torch.cuda.synchronize()
        te = time.perf_counter() - t0
        g.close()
        te = max_over_ranks(te * 1e3, device=dev) / 1e3
        # pinned host-to-device copy bandwidth of this process, measured on
        # the same buffers right after: the bound the upload puts on e2e
        probe_b = need[0]
        src = host["tok"][probe_b]
        dst = torch.empty_like(src, device=dev)
        def copy_gbps(a, reps):
            out = []
            for _ in range(reps):
                c0, c1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                c0.record()
                dst.copy_(a, non_blocking=True)
                c1.record()
                torch.cuda.synchronize()
                out.append(a.numel() * 4 / (c0.elapsed_time(c1) / 1e3) / 1e9)
            return out
        probe = copy_gbps(src, 5)
        best = max(probe)
        # the loop uploads each pinned buffer once; a buffer pinned now and
        # uploaded three times shows what a first upload costs
        try:
            fresh = torch.empty_like(src, pin_memory=True)
            fresh.copy_(tokens[:fresh.numel()])
            fresh_gbps = copy_gbps(fresh, 3)
            del fresh
        except Exception as ex:   # a diagnostic only
            fresh_gbps = str(ex)[:200]
        del dst
        e2e_val = job_throughput(ne, te * 1e3, world)
        bound = best * 1e9 / (h2d / Ke) * (ne / Ke) * world
        e2e = {"value": e2e_val, "unit": "req/s", "h2d_bytes_per_step": h2d // Ke,
               "d2h_bytes_per_step": d2h // Ke, "steps": Ke, "h2d_pinned_GBps": best,
               "h2d_bound_req_s": bound, "frac_of_h2d_bound": e2e_val / bound,
               "h2d_probe_GBps": probe, "h2d_fresh_buffer_GBps": fresh_gbps,
               "loop_upload_GBps": (h2d / Ke) / (te / Ke) / 1e9}

    # -- device-resident run -------------------------------------------------
    g = make_sched()
    for j in range(WP):
        step(g, j)
    torch.cuda.synchronize()
    assert g.last_error() == 0
    D.dm_get_stage_times(g.h, reset=True)
    D.dm_set_profiling(g.h, True, stages=["hash"])   # the hash+probe kernel only: events elsewhere cost time
    sampler = ClockSampler(local)
    time.sleep(0.3)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    wall0 = time.time()
    ev0.record()
    nreq = 0
    prompt_bytes = 0
    for j in range(WP, WP + K):
        nreq += step(g, j)
        b = j % used
        prompt_bytes += 4 * int(tr.L[tr.batches[b][0]:tr.batches[b][1]].sum())
    ev1.record()
    torch.cuda.synchronize()
    wall1 = time.time()
    if world > 1:
        dist.barrier()
    sampler.stop()
    ms = ev0.elapsed_time(ev1)
    st = D.dm_get_stage_times(g.h, reset=True)
    D.dm_set_profiling(g.h, False)
    err = g.last_error()
    assert err == 0, D.status_string(err)
    ms = max_over_ranks(ms, device=dev)
    value = job_throughput(nreq, ms, world)
    hash_ms, hash_calls = st["hash"]
    hash_avg_s = hash_ms / 1e3 / max(hash_calls, 1)
    bytes_per_launch = prompt_bytes / max(hash_calls, 1)
    peak, peak_kind = peaks()
    # hashing, ring lookup and probes run in one kernel: its event-timed
    # duration is the whole hash+probe path of the metric
    achieved = bytes_per_launch / hash_avg_s / 1e9
    prompt_gbps = achieved
    rebuilds, compactions = D.dm_get_maint_counts(g.h)   # over the warm-up and timed steps

    # per-stage breakdown: a fresh handle replays the same steps with every
    # stage timed (events between kernels stop their launch overlap, so this
    # run is not the headline)
    g.close()
    del g
    g = make_sched()
    cmp_batches = 0 if (args.no_cpu or rank != 0 or world != 1) else min(args.cpu_batches, used)
    gpu_out = {}   # the batches the CPU baseline routes: compared decision by decision below
    for j in range(WP):
        n = step(g, j)
        if j < cmp_batches:
            gpu_out[j] = g.results(n)
    D.dm_get_stage_times(g.h, reset=True)
    D.dm_set_profiling(g.h, True)
    for j in range(WP, WP + K):
        n = step(g, j)
        if j < cmp_batches:
            gpu_out[j] = g.results(n)
    st_all = D.dm_get_stage_times(g.h, reset=True)
    D.dm_set_profiling(g.h, False)
    assert g.last_error() == 0
    met, _ = D.dm_get_metrics(g.h)
    stage_ms = {k: v[0] / max(v[1], 1) for k, v in st_all.items()}
    # route: setup (with the queue drain), hash + ring lookup + probes (one
    # kernel), choice (with the segment carries) (3); commit: maint_a (with
    # the maintenance plan), maint_c (with the commit prep), commit_touch,
    # evict (4); rebalance (1)
    # (the cluster-wide rules add the carries and the all-instance probe kernels)
    launches_per_step = 3 + 4 + (1 if w.get("rebalance") else 0) + (2 if rule >= D.DM_RULE_LEAST_LOADED else 0)
    if args.adapt:   # window end: the update kernel, once per window
        launches_per_step += 1.0 / kw["adapt_window"]
    clocks = sampler.summary(wall0, wall1)
    g.close()
    del g

    # -- CPU oracle baseline (rank 0, N=1 only) ------------------------------------
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu:
        cb = list(range(min(args.cpu_batches, used)))

        def host_tokens(b):
            s, e, doff, dlen, nt, t0 = meta[b]
            return tokens[t0:t0 + nt].cpu().numpy().view(np.uint32)

        ora_out = {}
        extra = {"choice_rule": rule}
        if args.adapt:
            extra.update(adapt_step_blocks=kw["adapt_step_blocks"], adapt_max_blocks=kw["adapt_max_blocks"],
                         adapt_window=kw["adapt_window"])
        n_cpu, t_cpu = cpu_oracle_run(tr, w, [], cb, host_tokens, tr.max_instance_id(), keep=ora_out, extra=extra)
        # the GPU's decisions for the same batches must be the oracle's, bit for bit
        compared = 0
        for b in cb:
            if b not in gpu_out:
                continue
            for k, want in ora_out[b].items():
                got = gpu_out[b][k].astype(want.dtype)
                if not np.array_equal(got, want):
                    bad = np.nonzero(got != want)[0]
                    raise SystemExit(f"bench: GPU and oracle differ in batch {b}, {k} at {bad[:8].tolist()}")
            compared += len(ora_out[b]["chosen"])
        cpu = {"value": n_cpu / t_cpu, "unit": "req/s", "cores": 1, "kind": "oracle",
               "sample": f"first {len(cb)} batches ({n_cpu} requests) of the same trace, "
                         f"route+commit, {t_cpu:.1f} s",
               "decisions_compared": compared, "decisions_equal": True}

    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": "req/s", "n_gpus": world, "steps": K, "warmup": W,
            "ms_per_step": ms / K, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "u32 tokens / u64 integer arithmetic", "data": "synthetic",
            "prompt_GBps": prompt_gbps,
            "config": {"workload": f"{w['name']}: {w['n_instances']} instances x {w['vnodes']} vnodes, "
                                   f"batches of {w['batch']} prompts of {describe_lengths(w)} tokens "
                                   f"(~{bytes_per_launch / 1e6:.0f} MB per batch)",
                       "global_batch": w["batch"], "parallelism": f"replicas x{world}",
                       "cache_prefill_batches": P,
                       "choice_rule": args.rule,
                       "hash_prefix": (f"adaptive: base {w['route_prefix_blocks']} blocks, step {kw['adapt_step_blocks']}, "
                                       f"max {kw['adapt_max_blocks']}, window {kw['adapt_window']} batch(es)"
                                       if args.adapt else f"fixed {w['route_prefix_blocks']} blocks"),
                       "l2": ("inputs larger than L2 (each batch > 129 MB, distinct per step)"
                              if bytes_per_launch > 129e6 else
                              "batches smaller than L2, L2 not flushed between steps"),
                       "replay": "steps beyond the trace replay its batches cyclically" if WP + K > nb else "none"},
            "roofline": {"bound": "hbm", "kernel": "k_hash_probe (hashing + ring lookup + cache probes, one kernel)",
                         "achieved": achieved,
                         "peak": peak, "peak_kind": peak_kind, "unit": "GB/s", "frac": achieved / peak,
                         "traffic": traffic_per_launch(bytes_per_launch), "bytes_per_launch": bytes_per_launch,
                         "avg_launch_ms": hash_avg_s * 1e3},
            "stage_ms_per_step": stage_ms,
            "stage_note": "separate replay with every stage event-timed; hash = the hash+probe kernel",
            "serving": {"hit_rate": met["hit_tokens"] / max(met["prompt_tokens"], 1),
                        "cv_mean": met["cv_sum"] / max(met["cv_samples"], 1),
                        "slo_attainment": met["slo_met"] / max(met["completed"], 1),
                        "ttft_p50_us": met["ttft_p50_us"], "ttft_p90_us": met["ttft_p90_us"],
                        "completed": met["completed"], "requests": met["requests"],
                        "note": "scheduler time model over the stage-breakdown replay"},
            "e2e": e2e, "cpu_baseline": cpu, "gpu_launches": int(round(launches_per_step * K)), "clocks": clocks,
            "maintenance": {"index_rebuilds": rebuilds, "log_compactions": compactions,
                            "steps": WP + K, "note": "commits of the headline run that rebuilt an index or compacted a log"},
        }
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
