"""The debug build (libdualmap_debug.so, the sources compiled with
-DDM_DEBUG) on small traces against the CPU oracle: its device-side index
checks (segment and block offsets inside the batch scratch, ring search
results inside the ring, candidate ids inside the instance table, queue rows,
a commit segment's records inside the instance's log window) record
DM_ERR_BOUNDS instead of trapping.  Every decision must match the oracle and
no check may fire.  The traces run in a child process, which loads the debug
library (DM_LIBRARY=debug); a process loads only one of the two."""

import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)

CHILD = r"""
import sys
sys.path.insert(0, {root!r})
sys.path.insert(0, {tests!r})
from paper_2602_06502_gb300 import dualmap as D
assert D.LIB_PATH.endswith("libdualmap_debug.so"), D.LIB_PATH
from parity_harness import Pair, run_trace
from tracegen import Trace, workload

# eviction, log compaction, index rebuilds and rebalancing on a small cache
w = workload("tiny", n_requests=2000, batch=100, capacity=700, zipf_s=1.3, rho=1.2)
p = Pair(w, max_touch=2600)
run_trace(p, Trace(w), rebalance=True, state_every=5)
assert D.dm_last_error(p.gpu.h) == D.DM_OK
# tails past the routing head, the SLO switch, 4,096-prompt batches
tr = Trace(workload("agent", n_requests=3 * 4096))
p = Pair(tr.cfg, max_batch_tokens=40_000_000, max_touch=1 << 20)
run_trace(p, tr)
assert D.dm_last_error(p.gpu.h) == D.DM_OK
# long prompts (runs past the routing head's first blocks), two batches
tr = Trace(workload("longctx", n_requests=2 * 512))
p = Pair(tr.cfg, max_batch_tokens=70_000_000, max_touch=1 << 20, capacity=200_000)
run_trace(p, tr)
assert D.dm_last_error(p.gpu.h) == D.DM_OK
print("debug build: parity and no bounds error")
"""


def test_debug_build_matches_the_oracle_and_no_index_check_fires():
    from paper_2602_06502_gb300 import build as B
    B.build(debug=True)
    env = dict(os.environ, DM_LIBRARY="debug")
    r = subprocess.run([sys.executable, "-c", CHILD.format(root=ROOT, tests=HERE)], env=env, capture_output=True,
                       text=True, timeout=1500)
    assert r.returncode == 0, r.stdout[-4000:] + r.stderr[-4000:]
    assert "no bounds error" in r.stdout
