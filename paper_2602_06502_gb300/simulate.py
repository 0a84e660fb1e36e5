"""Replay a synthetic trace under each choice rule and report the serving
metrics the paper compares schedulers by: cache hit rate and load-balance CV
(Sec. 2.2), SLO attainment and TTFT percentiles (Sec. 4.1), under the
scheduler's own time model (each instance runs its queued prefill work at
one microsecond per microsecond from the batch times on).

Every step runs in the library's kernels through the C ABI; this module only
generates the trace, calls the library and formats the result:

    python -m paper_2602_06502_gb300.simulate --workload tiny --set rho=0.9
    python -m paper_2602_06502_gb300.simulate --workload agent --rules dualmap,least_loaded,min_ttft

One JSON line per rule.  The cluster-wide rules probe every live instance
for every request, which the two-candidate rules avoid; the choice stage's
time per batch is reported beside the metrics.
"""

import argparse
import json
import os
import sys

import numpy as np


def simulate(workload_name, rules, overrides=None, rebalance=None, batches=None, device="cuda:0", adapt=None):
    """Replay the trace once per rule; returns one dict per rule."""
    import torch

    sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
    import tracegen.device as TD
    from tracegen import Trace, workload

    from . import dualmap as D
    from .scheduler import Scheduler

    w = workload(workload_name, **(overrides or {}))
    tr = Trace(w)
    nb = len(tr.batches) if batches is None else min(batches, len(tr.batches))
    if rebalance is None:
        rebalance = bool(w.get("rebalance"))
    dev = torch.device(device)
    ntok = int(tr.req_off[tr.batches[nb - 1][1]])
    tokens = torch.empty(ntok + 4, dtype=torch.int32, device=dev)
    TD.fill_range(tr, 0, tr.batches[nb - 1][1], tokens[:ntok])
    max_id = tr.max_instance_id()
    max_len = int(max(tr.batch_layout(b)[4] for b in range(nb)))
    events = {}
    for b, kind, i in tr.events:
        events.setdefault(b, []).append((kind, i))
    out = []
    for name in rules:
        rule = D.RULE_NAMES.index(name)
        g = Scheduler(block_tokens=w["block_tokens"], route_prefix_blocks=w["route_prefix_blocks"],
                      vnodes=w["vnodes"], max_instances=max_id + 1, capacity=w["capacity"], slo_us=w["slo_us"],
                      cost_us=w["cost_us"], max_batch=w["batch"], max_batch_tokens=max(max_len, 1 << 16),
                      seed=w["seed"], choice_rule=rule, device=device, **(adapt or {}))
        for i in range(w["n_instances"]):
            assert g.add_instance(i) == 0
        D.dm_set_profiling(g.h, True, stages=["choice"])
        ksum = kmax = 0
        for b in range(nb):
            for kind, i in events.get(b, []):
                assert (g.add_instance(i) if kind == "add" else g.remove_instance(i)) == 0
            s, e, off, lens, nt = tr.batch_layout(b)
            t0 = int(tr.req_off[s])
            g.route(tokens[t0:t0 + nt + 4], torch.from_numpy(off.view(np.int64)).to(dev),
                    torch.from_numpy(lens.view(np.int32)).to(dev), e - s, nt, tr.batch_time(b))
            K = g.route_blocks(e - s)
            ksum += int(K.sum())
            kmax = max(kmax, int(K.max()))
            if rebalance:
                g.rebalance()
            g.commit()
        err = g.last_error()
        if err:
            raise D.DualMapError(err, f"rule {name}")
        m, _ = D.dm_get_metrics(g.h)
        tree = D.dm_export_prefix_tree(g.h)
        st = D.dm_get_stage_times(g.h)
        g.close()
        ms, calls = st["choice"]
        out.append({
            "rule": name, "workload": w["name"], "batches": nb, "requests": m["requests"],
            "hit_rate": m["hit_tokens"] / max(m["prompt_tokens"], 1),
            "cv_mean": m["cv_sum"] / max(m["cv_samples"], 1),
            "slo_attainment": m["slo_met"] / max(m["completed"], 1),
            "est_slo_attainment": m["est_slo_met"] / max(m["requests"], 1),
            "completed": m["completed"], "ttft_mean_us": m["ttft_sum_us"] / max(m["completed"], 1),
            "ttft_p50_us": m["ttft_p50_us"], "ttft_p90_us": m["ttft_p90_us"], "ttft_p99_us": m["ttft_p99_us"],
            "switched": m["switched"], "choice_ms_per_batch": ms / max(calls, 1),
            "hash_blocks_mean": ksum / max(m["requests"], 1), "hash_blocks_max": kmax,
            "prefix_tree_nodes": None if not adapt else len(tree),
        })
    return out


def main():
    from . import dualmap as D
    ap = argparse.ArgumentParser(description=__doc__.split("\n\n")[0])
    ap.add_argument("--workload", default="tiny")
    ap.add_argument("--rules", default="all", help="comma-separated rule names, or all")
    ap.add_argument("--set", action="append", default=[], metavar="KEY=VALUE", help="override a workload field")
    ap.add_argument("--rebalance", choices=["auto", "on", "off"], default="auto")
    ap.add_argument("--batches", type=int, default=None)
    ap.add_argument("--adapt", default="", metavar="STEP,MAX[,WINDOW]",
                    help="adaptive hash-prefix length (blocks per step, longest prefix, batches per window)")
    args = ap.parse_args()
    rules = D.RULE_NAMES if args.rules == "all" else args.rules.split(",")
    over = {}
    for kv in args.set:
        k, v = kv.split("=", 1)
        over[k] = float(v) if "." in v else int(v)
    rb = None if args.rebalance == "auto" else args.rebalance == "on"
    ad = None
    if args.adapt:
        a = [int(x) for x in args.adapt.split(",")]
        ad = dict(adapt_step_blocks=a[0], adapt_max_blocks=a[1], adapt_window=a[2] if len(a) > 2 else 1)
    for r in simulate(args.workload, rules, over, rb, args.batches, adapt=ad):
        print(json.dumps(r), flush=True)


if __name__ == "__main__":
    main()
