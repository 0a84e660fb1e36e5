"""Synthetic workload shapes for the DualMap routing path.

The paper evaluates on the Mooncake *Conversation* and *Tool&Agent* traces
(Appendix A.2.1, Table "workload-characteristics"); those traces are not
available, so every workload here is a seeded synthetic stand-in with the
shape described below.  Nothing in this module computes any part of the
routing method: it only fixes sizes, distributions and seeds.

Each workload is a plain dict.  Keys:
  name, n_instances, vnodes, block_tokens, route_prefix_blocks, capacity,
  slo_us, cost_us, n_requests, batch, vocab, rho, kind (+ kind-specific keys),
  rebalance (bool), scale_every (0 = no add/remove events), seed.
"""

import copy

WORKLOADS = {
    # Tiny trace: 8 instances, 2,000 requests of 128-2,048 tokens, 50 shared
    # prefixes (Zipf s=1.0, 256-1,024 tokens) + unique suffix.
    "tiny": dict(
        name="tiny", kind="prefix_suffix",
        n_instances=8, vnodes=64, block_tokens=16, route_prefix_blocks=16,
        capacity=65536, slo_us=2_000_000, cost_us=1,
        n_requests=2000, batch=256, vocab=32000, rho=0.6,
        len_lo=128, len_hi=2048, n_prefix=50, zipf_s=1.0,
        prefix_lo=256, prefix_hi=1024,
        rebalance=False, scale_every=0, seed=1001,
    ),
    # Multi-turn conversation: 32 instances, 10,000 concurrently active
    # sessions, Geom(0.2) turns capped at 20, each turn = whole history +
    # 50-500 new tokens, prompt capped at 16,384 tokens, vocab 128,000.
    "multiturn": dict(
        name="multiturn", kind="sessions",
        n_instances=32, vnodes=256, block_tokens=16, route_prefix_blocks=16,
        capacity=1 << 20, slo_us=2_000_000, cost_us=1,
        n_requests=100_000, batch=1024, vocab=128_000, rho=0.7,
        n_sessions=10_000, turn_p=0.2, max_turns=20,
        chunk_lo=50, chunk_hi=500, max_prompt=16_384,
        rebalance=False, scale_every=0, seed=1002,
    ),
    # Agent / tool: 64 instances, 1M requests = one of 200 system-prompt
    # templates (2,048-8,192 tokens, Zipf s=1.2) + 100-1,000 unique tokens;
    # tight load so the SLO switch fires often.
    "agent": dict(
        name="agent", kind="template",
        n_instances=64, vnodes=256, block_tokens=16, route_prefix_blocks=16,
        capacity=1 << 20, slo_us=1_000_000, cost_us=1,
        n_requests=1_000_000, batch=4096, vocab=32000, rho=1.0,
        n_prefix=200, zipf_s=1.2, prefix_lo=2048, prefix_hi=8192,
        uniq_lo=100, uniq_hi=1000,
        rebalance=False, scale_every=0, seed=1003,
    ),
    # Long-context bandwidth stress: 128 instances, 65,536 requests of
    # 32,768-131,072 tokens (~21.5 GB of token IDs), 64 shared 16k-token
    # prefixes (Zipf s=0.8) + unique remainder, batches of 512.
    "longctx": dict(
        name="longctx", kind="fixed_prefix",
        n_instances=128, vnodes=256, block_tokens=16, route_prefix_blocks=16,
        capacity=1 << 20, slo_us=2_000_000, cost_us=1,
        n_requests=65_536, batch=512, vocab=32000, rho=0.5,
        len_lo=32_768, len_hi=131_072, n_prefix=64, zipf_s=0.8,
        prefix_len=16_384,
        rebalance=False, scale_every=0, seed=1004,
    ),
    # Scaling + hotspot: 256 instances with 1,024 vnodes each, 2M requests of
    # 512-8,192 tokens over 1,000 prefixes (Zipf s=1.4), an instance added or
    # removed every 100k requests, rebalancing after every 4,096-request batch.
    "scaling": dict(
        name="scaling", kind="prefix_suffix",
        n_instances=256, vnodes=1024, block_tokens=16, route_prefix_blocks=16,
        capacity=262_144, slo_us=1_000_000, cost_us=1,
        n_requests=2_000_000, batch=4096, vocab=32000, rho=0.9,
        len_lo=512, len_hi=8192, n_prefix=1000, zipf_s=1.4,
        prefix_lo=256, prefix_hi=2048,
        rebalance=True, scale_every=100_000, seed=1005,
    ),
}

ORDER = ["tiny", "multiturn", "agent", "longctx", "scaling"]


def workload(name, **overrides):
    """A copy of workload `name` with keyword overrides applied."""
    w = copy.deepcopy(WORKLOADS[name])
    for k, v in overrides.items():
        if k not in w:
            raise KeyError(f"unknown workload key {k!r}")
        w[k] = v
    return w
