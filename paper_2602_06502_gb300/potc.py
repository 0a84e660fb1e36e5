"""The maximum-load sweep of App. A.8 ("Optimal Candidate Set Size") on the
GPU: for each cluster size n and candidate count d, `trials` trials of
m = balls_per_bin * n balls placed by the power of d choices
(dm_potc_max_loads), reporting the maximum load deviation (maximum bin load
minus m/n): mean, median and 99th percentile over the trials, and the
kernel time.

    python -m paper_2602_06502_gb300.potc --n 8,16,24,32 --d 1,2,3,4 --trials 10000
"""

import argparse
import json

import numpy as np


def sweep(ns, ds, trials, balls_per_bin=1000, seed=2602):
    import torch

    from . import dualmap as D

    out = torch.zeros(trials, dtype=torch.int32, device="cuda")
    rows = []
    for n in ns:
        m = balls_per_bin * n
        for d in ds:
            ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            stream = torch.cuda.current_stream().cuda_stream
            ev0.record()
            rc = D.dm_potc_max_loads(n, m, d, trials, seed + 1000 * n + d, out, stream)
            ev1.record()
            if rc:
                raise D.DualMapError(rc, "dm_potc_max_loads")
            torch.cuda.synchronize()
            dev = out.cpu().numpy().astype(np.int64) - balls_per_bin
            rows.append({"n": n, "d": d, "m": m, "trials": trials, "dev_mean": float(dev.mean()),
                         "dev_median": float(np.median(dev)), "dev_p99": float(np.percentile(dev, 99)),
                         "kernel_ms": ev0.elapsed_time(ev1),
                         "balls_per_s": trials * m / (ev0.elapsed_time(ev1) / 1e3)})
    return rows


def main():
    ap = argparse.ArgumentParser(description=__doc__.split("\n\n")[0])
    ap.add_argument("--n", default="8,16,24,32")
    ap.add_argument("--d", default="1,2,3,4")
    ap.add_argument("--trials", type=int, default=10000)
    ap.add_argument("--balls-per-bin", type=int, default=1000)
    args = ap.parse_args()
    for r in sweep([int(x) for x in args.n.split(",")], [int(x) for x in args.d.split(",")], args.trials,
                   args.balls_per_bin):
        print(json.dumps(r), flush=True)


if __name__ == "__main__":
    main()
