"""Pins of the oracle's adaptive hash-prefix length (Sec. 3.2, "how long
prefix is appropriate"): a node of the prefix hotness tree is a prefix
identified by its last block's key; a request walks from K_route blocks,
one step deeper while its node is expanded; at the end of each window a node
whose share of the window's requests exceeds 2/n is expanded and an expanded
node whose share falls below 1/n is dropped (n = live instances).  Expected
values are worked out by hand from that rule."""

import numpy as np
import pytest

from oracle import oracle as O

B, KR, STEP = 16, 4, 4


def mk(n=4, kmax=40, window=1, kroute=KR, step=STEP, M=None):
    o = O.Oracle(block_tokens=B, route_prefix_blocks=kroute, vnodes_per_instance=16, max_instances=M or n + 2,
                 cache_capacity_blocks=1 << 16, slo_us=10**9, cost_us_per_token=1, hot_num=3, hot_den=2,
                 max_batch=64, max_batch_tokens=1 << 20, seed=11, adapt_step_blocks=step,
                 adapt_max_blocks=kmax, adapt_window=window)
    for i in range(n):
        assert o.add_instance(i) == 0
    return o


RNG = np.random.default_rng(7)
PREFIX_A = RNG.integers(0, 32000, 200, dtype=np.uint32)   # blocks 0..11 whole, block 12 half


def a_prompt(L=400):
    return np.concatenate([PREFIX_A, RNG.integers(0, 32000, L - len(PREFIX_A), dtype=np.uint32)])


def u_prompt(L=400):
    return RNG.integers(0, 32000, L, dtype=np.uint32)


class Run:
    def __init__(self, o):
        self.o, self.t = o, 0

    def batch(self, prompts):
        lens = np.array([len(p) for p in prompts], np.uint32)
        off = np.zeros(len(prompts), np.uint64)
        acc = 0
        for i, p in enumerate(prompts):
            off[i] = acc
            acc += (len(p) + 3) // 4 * 4
        tok = np.zeros(acc + 4, np.uint32)
        for i, p in enumerate(prompts):
            tok[int(off[i]):int(off[i]) + len(p)] = p
        self.t += 1000
        rc, out = self.o.route_batch(tok, off, lens, self.t)
        assert rc == 0
        assert self.o.commit() == 0
        return self.o.route_blocks(), out


def mixed(n_a, n_u):
    return [a_prompt() for _ in range(n_a)] + [u_prompt() for _ in range(n_u)]


def test_hot_prefix_deepens_one_step_per_window_until_requests_diverge():
    """n = 4, 6 of 10 requests share a 200-token prefix (12 whole blocks):
    share 0.6 > 2/4, so the node deepens 4 -> 8 -> 12 -> 16 blocks; at 16
    blocks every request's node differs (block 12 holds its own tokens),
    so the walk stops there."""
    r = Run(mk())
    seen = []
    for _ in range(5):
        K, _ = r.batch(mixed(6, 4))
        assert K[6:].tolist() == [KR] * 4
        assert len(set(K[:6].tolist())) == 1
        seen.append(int(K[0]))
    assert seen == [4, 8, 12, 16, 16]
    assert len(r.o.prefix_tree()) == 3          # nodes at 4, 8 and 12 blocks


def test_cold_prefix_collapses_and_unreached_nodes_drop():
    """After the tree holds A's nodes at 4, 8, 12, a window where 1 of 10
    requests has prefix A (share 0.1 < 1/4) drops all three."""
    r = Run(mk())
    for _ in range(4):
        r.batch(mixed(6, 4))
    assert len(r.o.prefix_tree()) == 3
    K, _ = r.batch(mixed(1, 9))
    assert K[0] == 16                            # still walks the old tree this batch
    assert len(r.o.prefix_tree()) == 0
    K, _ = r.batch(mixed(1, 9))
    assert K[0] == KR


def test_hysteresis_between_one_and_two_over_n():
    """Share 3/10 with n = 4 is neither > 2/4 nor < 1/4: an expanded node
    stays expanded and a leaf is not expanded."""
    r = Run(mk())
    r.batch(mixed(6, 4))                         # expands A at 4 blocks
    tree = r.o.prefix_tree().tolist()
    K, _ = r.batch(mixed(3, 7))                  # A walks to 8; node 8 reached by 3 of 10
    assert K[0] == 8
    assert r.o.prefix_tree().tolist() == tree    # node 4 kept, node 8 not expanded
    K, _ = r.batch(mixed(3, 7))
    assert K[0] == 8


@pytest.mark.parametrize("n,n_a,expand", [(4, 5, False), (4, 6, True), (5, 4, False), (5, 5, True)])
def test_expansion_threshold_is_strict(n, n_a, expand):
    """Expand iff count * n > 2 T (T = 10): 5 * 4 = 20 is not > 20; 4 * 5 =
    20 is not > 20."""
    r = Run(mk(n=n))
    r.batch(mixed(n_a, 10 - n_a))
    assert (len(r.o.prefix_tree()) == 1) == expand


def test_shrink_threshold_is_strict():
    """Drop iff count * n < T: with n = 5 and T = 10, 2 requests (10) keep
    the node, 1 request (5) drops it."""
    r = Run(mk(n=5))
    r.batch(mixed(6, 4))
    assert len(r.o.prefix_tree()) == 1
    r.batch(mixed(2, 8))                         # node 4: 2 * 5 = 10, not < 10
    assert len(r.o.prefix_tree()) == 1
    r.batch(mixed(1, 9))
    assert len(r.o.prefix_tree()) == 0


def test_cap_on_prefix_length():
    """adapt_max_blocks = 10: the walk goes 4 -> 8 -> 10 and a node at the
    cap is never expanded."""
    r = Run(mk(kmax=10))
    seen = [int(r.batch(mixed(6, 4))[0][0]) for _ in range(4)]
    assert seen == [4, 8, 10, 10]
    assert len(r.o.prefix_tree()) == 2


def test_window_of_two_batches():
    """Counts cover the whole window: 6 of 10 then 0 of 10 is 6 of 20 (6 * 4
    = 24, not > 40): nothing expands, whereas a one-batch window expands
    after the first batch."""
    for window, want in ((1, 8), (2, 4)):
        r = Run(mk(window=window))
        r.batch(mixed(6, 4))
        K, _ = r.batch(mixed(1, 9))
        assert K[0] == want
    r = Run(mk(window=2))
    r.batch(mixed(6, 4))
    r.batch(mixed(6, 4))                         # 12 of 20: 48 > 40
    K, _ = r.batch(mixed(1, 9))
    assert K[0] == 8


def test_threshold_uses_live_instances():
    """With 4 live instances 6 of 10 is hot (24 > 20); after removing one (n
    = 3: 18 is not > 20) it is not."""
    for remove, want in ((False, 1), (True, 0)):
        o = mk(n=4)
        if remove:
            assert o.remove_instance(3) == 0
        r = Run(o)
        r.batch(mixed(6, 4))
        assert len(o.prefix_tree()) == want


def test_short_prompts_and_positions_equal_fixed_length_hash():
    """A prompt shorter than K_route hashes all its blocks; a request walked
    to K blocks gets the ring owner of the position a fixed-length hash of K
    blocks gives (same seed: same key material)."""
    r = Run(mk())
    K, _ = r.batch([u_prompt(40)] + mixed(6, 3))
    assert K[0] == 2                             # 40 tokens: 2 whole blocks
    prompts = mixed(6, 4)
    K, out = r.batch(prompts)
    assert K[0] == 8
    fixed = O.Oracle(block_tokens=B, route_prefix_blocks=8, vnodes_per_instance=16, max_instances=6,
                     cache_capacity_blocks=1 << 16, slo_us=10**9, cost_us_per_token=1, hot_num=3, hot_den=2,
                     max_batch=64, max_batch_tokens=1 << 20, seed=11)
    _, pos = fixed.prompt_keys(prompts[0])
    assert r.o.ring_owners(pos[:1], 0)[0] == out["cand1"][0]
    raw2 = r.o.ring_owners(pos[1:], 1)[0]
    assert out["cand2"][0] == (raw2 if raw2 != out["cand1"][0] else r.o.next_live(int(out["cand1"][0])))


def test_no_hot_prefix_is_fixed_length_routing():
    """Batches of unrelated prompts never make a node hot: every output
    equals routing with the fixed K_route, and the tree stays empty."""
    a, b = Run(mk()), Run(mk(step=0))
    for _ in range(4):
        prompts = [u_prompt(int(L)) for L in RNG.integers(16, 600, 12)]
        Ka, oa = a.batch(prompts)
        Kb, ob = b.batch(prompts)
        assert Ka.tolist() == Kb.tolist()
        for k in oa:
            assert np.array_equal(oa[k], ob[k]), k
    assert len(a.o.prefix_tree()) == 0


def test_identical_prefixes_share_length_and_candidates():
    """Requests with the same first K blocks walk the same nodes, so they get
    the same length and the same candidate pair: identical prefixes still map
    to one candidate pair with adaptive lengths."""
    r = Run(mk())
    for _ in range(3):
        K, out = r.batch(mixed(6, 4))
        assert len(set(K[:6].tolist())) == 1
        assert len(set(zip(out["cand1"][:6].tolist(), out["cand2"][:6].tolist()))) == 1


def test_bad_adaptive_config_rejected():
    with pytest.raises(ValueError):
        mk(kmax=KR)                              # cap not above K_route
    with pytest.raises(ValueError):
        mk(kmax=4096)                            # above 2048
    with pytest.raises(ValueError):
        mk(window=0)


@pytest.mark.parametrize("window", [1, 3])
def test_matches_an_independent_tree_model_on_a_trace(window):
    """The hotness tree re-implemented in plain Python (walk, per-window node
    counts, expand above 2T/n, drop below T/n) on a Zipf-skewed trace: every
    request's length and the expanded set after every batch agree."""
    from tracegen import Trace, workload
    w = workload("tiny", n_requests=1500, batch=100, zipf_s=1.2)
    tr = Trace(w)
    kr, step, kmax, n = w["route_prefix_blocks"], 8, 96, w["n_instances"]
    o = O.Oracle(**O.config_from_workload(w, max_instances=n), adapt_step_blocks=step, adapt_max_blocks=kmax,
                 adapt_window=window)
    for i in range(n):
        assert o.add_instance(i) == 0
    expanded, counts, T, nb = set(), {}, 0, 0
    deepest = 0
    for b in range(len(tr.batches)):
        s, e, off, lens, nt = tr.batch_layout(b)
        tok = tr.batch_tokens(b)
        want = []
        for r in range(len(lens)):
            keys = o.prompt_keys(tok[int(off[r]):int(off[r]) + int(lens[r])])[0].tolist()
            nblk = len(keys)
            d = min(kr, nblk)
            path = [(keys[d - 1], d)]
            while d < nblk and d < kmax and keys[d - 1] in expanded:
                d = min(d + step, nblk, kmax)
                path.append((keys[d - 1], d))
            want.append(d)
            for k, dep in path:
                c, _ = counts.get(k, (0, dep))
                counts[k] = (c + 1, dep)
        rc, out = o.route_batch(tok, off, lens, tr.batch_time(b))
        assert rc == 0
        assert o.route_blocks().tolist() == want, b
        T += len(lens)
        nb += 1
        if nb == window:
            keep = {k for k in expanded if not counts.get(k, (0, 0))[0] * n < T}
            new = {k for k, (c, dep) in counts.items() if k not in expanded and dep < kmax and c * n > 2 * T}
            expanded, counts, T, nb = keep | new, {}, 0, 0
        assert sorted(expanded) == o.prefix_tree().tolist(), b
        deepest = max(deepest, max(want))
        assert o.commit() == 0
    assert deepest > kr                          # the trace does make prefixes hot
