"""The rule-comparison simulator (paper_2602_06502_gb300.simulate) on the GPU:
its metrics for every rule equal the oracle's replay of the same trace, and
the cluster-wide rules order as Sec. 2.2 reports."""

import pytest

from oracle import oracle as O
from parity_harness import lib_ready
from tracegen import Trace, workload

pytestmark = pytest.mark.gpu

OVER = dict(n_requests=2000, batch=100, zipf_s=1.2, rho=0.9)


@pytest.fixture(scope="module", autouse=True)
def _built():
    lib_ready()


def _oracle(rule):
    w = workload("tiny", **OVER)
    tr = Trace(w)
    o = O.Oracle(**O.config_from_workload(w, max_instances=w["n_instances"]), choice_rule=rule)
    for i in range(w["n_instances"]):
        assert o.add_instance(i) == 0
    for b in range(len(tr.batches)):
        s, e, off, lens, nt = tr.batch_layout(b)
        assert o.route_batch(tr.batch_tokens(b), off, lens, tr.batch_time(b))[0] == 0
        assert o.commit() == 0
    return o.metrics()[0]


def test_simulator_matches_oracle_and_sec_2_2():
    from paper_2602_06502_gb300 import dualmap as D
    from paper_2602_06502_gb300.simulate import simulate
    res = {r["rule"]: r for r in simulate("tiny", D.RULE_NAMES, OVER)}
    for k, name in enumerate(D.RULE_NAMES):
        om = _oracle(k)
        r = res[name]
        assert r["requests"] == om["requests"] == 2000
        assert r["completed"] == om["completed"]
        assert r["hit_rate"] == om["hit_tokens"] / om["prompt_tokens"]
        assert r["cv_mean"] == om["cv_sum"] / om["cv_samples"]
        assert r["ttft_p90_us"] == om["ttft_p90_us"]
        assert r["choice_ms_per_batch"] > 0
    h = {k: v["hit_rate"] for k, v in res.items()}
    cv = {k: v["cv_mean"] for k, v in res.items()}
    assert h["cache_affinity"] > h["least_loaded"] and cv["least_loaded"] < cv["cache_affinity"]
    for r in ("min_ttft", "preble"):
        assert h["least_loaded"] < h[r] < h["cache_affinity"]
        assert cv["least_loaded"] < cv[r] < cv["cache_affinity"]
