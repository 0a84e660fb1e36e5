"""Pins of the oracle's routing with d candidates instead of two (App. A.8,
"Optimal Candidate Set Size"): d = 2 is DualMap's routing exactly, d = 1 is
cache affinity (the ring-1 owner, Sec. 1), the key material of functions
3..d continues DualMap's SplitMix64 stream (recomputed here from the
published generator), every ring position and candidate against a plain
recomputation (NH, fmix64, linear ring scan, the distinct rule), the d-way
choice against a plain-Python model of the rule and of the loads, the
cache-affinity guarantee of Sec. 2.3 for d candidates, and the load
spread App. A.8 argues from (many more requests on the busiest instance
with one choice than with two)."""

import numpy as np
import pytest

from oracle import oracle as O
from tracegen import Trace, workload

M64 = (1 << 64) - 1


def sm64(state):
    """SplitMix64 (Steele, Lea, Flood 2014): (new state, output)."""
    state = (state + 0x9E3779B97F4A7C15) & M64
    z = state
    z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & M64
    z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & M64
    return state, z ^ (z >> 31)


def fmix(k):
    """MurmurHash3's 64-bit finaliser."""
    k ^= k >> 33
    k = (k * 0xFF51AFD7ED558CCD) & M64
    k ^= k >> 33
    k = (k * 0xC4CEB9FE1A85EC53) & M64
    return k ^ (k >> 33)


def nh(block, K):
    return sum(((int(block[2 * i]) + int(K[2 * i])) & 0xFFFFFFFF) *
               ((int(block[2 * i + 1]) + int(K[2 * i + 1])) & 0xFFFFFFFF) for i in range(len(block) // 2)) & M64


def mk(d, M=12, V=16, C=1 << 16, slo=10**6, B=16, K=4, seed=11, live=None, rule=0):
    o = O.Oracle(block_tokens=B, route_prefix_blocks=K, vnodes_per_instance=V, max_instances=M,
                 cache_capacity_blocks=C, slo_us=slo, cost_us_per_token=1, hot_num=3, hot_den=2, max_batch=4096,
                 max_batch_tokens=1 << 30, seed=seed, candidates=d, choice_rule=rule)
    for i in (range(M) if live is None else live):
        assert o.add_instance(i) == 0
    return o


def tiny_trace(**kw):
    base = dict(n_requests=600, batch=100)
    base.update(kw)
    return Trace(workload("tiny", **base))


def test_key_material_continues_dualmaps_stream():
    B, seed = 16, 11
    o = mk(6, B=B, seed=seed)
    K1, K2, sc = o.key_material()
    st = seed
    draws = []
    for _ in range(2 * B + 7 + 4 * (B + 3)):
        st, z = sm64(st)
        draws.append(z)
    assert [int(x) for x in K1] == [z & 0xFFFFFFFF for z in draws[:B]]
    assert [int(x) for x in K2] == [z & 0xFFFFFFFF for z in draws[B:2 * B]]
    for f in range(6):
        Kf, s3 = o.key_material_f(f)
        if f < 2:
            want_K = K1 if f == 0 else K2
            want = [int(sc[f]), int(sc[3 + f]), int(sc[5 + f])]   # G_f, S_rf, S_vf
        else:
            base = 2 * B + 7 + (f - 2) * (B + 3)
            want_K = [z & 0xFFFFFFFF for z in draws[base:base + B]]
            want = [draws[base + B] | 1, draws[base + B + 1], draws[base + B + 2]]
        assert [int(x) for x in Kf] == [int(x) for x in want_K], f
        assert [int(x) for x in s3] == want, f


def test_positions_and_candidates_against_plain_recomputation():
    d, B, Kr = 5, 16, 4
    o = mk(d, M=9, V=12, B=B, K=Kr, live=[0, 1, 2, 4, 5, 7, 8])
    live = sorted({0, 1, 2, 4, 5, 7, 8})
    rng = np.random.default_rng(4)
    n = 60
    lens = rng.integers(B, 12 * B, size=n).astype(np.uint32)
    lens[:5] = B
    off = np.zeros(n, np.uint64)
    off[1:] = np.cumsum(lens[:-1].astype(np.uint64))
    tok = rng.integers(0, 1 << 32, size=int(lens.sum()), dtype=np.uint64).astype(np.uint32)
    tok[int(off[10]):int(off[10]) + int(lens[10])] = tok[int(off[11]):int(off[11]) + int(lens[10])] \
        if lens[11] >= lens[10] else tok[int(off[10]):int(off[10]) + int(lens[10])]
    rc, out = o.route_batch_d(d, tok, off, lens, 100)
    assert rc == 0
    rings = [o.ring(f) for f in range(d)]
    for r in range(n):
        p = tok[int(off[r]):int(off[r]) + int(lens[r])]
        nblk = len(p) // B
        K = min(Kr, nblk)
        cands = []
        for f in range(d):
            Kf, (G, Sr, Sv) = o.key_material_f(f)
            P = 0
            for k in range(K):
                P = (P + fmix((nh(p[k * B:(k + 1) * B], Kf) + (k + 1) * int(G)) & M64)) & M64
            pos = fmix(P ^ int(Sr))
            assert o.ring_position(p, f) == pos
            vp, ow, _ = rings[f]
            idx = [i for i in range(len(vp)) if int(vp[i]) >= pos]
            owner = int(ow[min(idx, key=lambda i: (int(vp[i]), i))] if idx else ow[0])
            while owner in cands:   # taken: the next live id after it, cyclically
                owner = live[(live.index(owner) + 1) % len(live)]
            cands.append(owner)
        assert out["cand"][r].tolist() == cands, r
        assert len(set(cands)) == d


def test_two_candidates_are_dualmaps_routing():
    tr = tiny_trace(zipf_s=1.2, rho=1.1)
    w = tr.cfg
    a = O.Oracle(**O.config_from_workload(w, candidates=2, slo_us=20_000))
    b = O.Oracle(**O.config_from_workload(w, candidates=2, slo_us=20_000))
    for i in range(w["n_instances"]):
        a.add_instance(i)
        b.add_instance(i)
    switched = 0
    for bi in range(len(tr.batches)):
        s, e, off, lens, _ = tr.batch_layout(bi)
        tok = tr.batch_tokens(bi)
        rc, want = a.route_batch(tok, off, lens, tr.batch_time(bi))
        rc2, got = b.route_batch_d(2, tok, off, lens, tr.batch_time(bi))
        assert rc == 0 and rc2 == 0
        assert np.array_equal(got["cand"][:, 0], want["cand1"]) and np.array_equal(got["cand"][:, 1], want["cand2"])
        assert np.array_equal(got["hit"][:, 0], want["hit1"]) and np.array_equal(got["hit"][:, 1], want["hit2"])
        assert np.array_equal(got["ttft"][:, 0], want["ttft1"]) and np.array_equal(got["ttft"][:, 1], want["ttft2"])
        assert np.array_equal(got["chosen"], want["chosen"]) and np.array_equal(got["switched"], want["switched"])
        switched += int(want["switched"].sum())
        a.commit()
        b.commit()
        assert np.array_equal(a.loads(), b.loads())
    assert switched > 0
    ma, mb = a.metrics()[0], b.metrics()[0]
    assert ma == mb


def test_one_candidate_is_cache_affinity():
    tr = tiny_trace(zipf_s=1.0)
    w = tr.cfg
    a = O.Oracle(**O.config_from_workload(w, choice_rule=O.RULE_GLOBAL_CACHE_AFFINITY))
    b = O.Oracle(**O.config_from_workload(w, candidates=2))
    for i in range(w["n_instances"]):
        a.add_instance(i)
        b.add_instance(i)
    for bi in range(len(tr.batches)):
        s, e, off, lens, _ = tr.batch_layout(bi)
        tok = tr.batch_tokens(bi)
        rc, want = a.route_batch(tok, off, lens, tr.batch_time(bi))
        rc2, got = b.route_batch_d(1, tok, off, lens, tr.batch_time(bi))
        assert rc == 0 and rc2 == 0
        assert np.array_equal(got["chosen"], got["cand"][:, 0])
        assert np.array_equal(got["chosen"], want["chosen"])
        assert not got["switched"].any()
        a.commit()
        b.commit()
        assert np.array_equal(a.loads(), b.loads())


@pytest.mark.parametrize("d", [3, 4])
def test_d_way_choice_matches_a_plain_model(d):
    """The oracle's choices and loads against the rule recomputed request
    by request from its reported candidates and hits, with the loads kept
    here (start of batch: the oracle's loads after the drain)."""
    tr = tiny_trace(zipf_s=1.3, rho=1.4, n_requests=800)
    w = tr.cfg
    o = O.Oracle(**O.config_from_workload(w, candidates=d, slo_us=30_000))
    for i in range(w["n_instances"]):
        o.add_instance(i)
    slo, switched = 30_000, 0
    for bi in range(len(tr.batches)):
        s, e, off, lens, _ = tr.batch_layout(bi)
        tok = tr.batch_tokens(bi)
        rc, got = o.route_batch_d(d, tok, off, lens, tr.batch_time(bi))
        assert rc == 0
        W = {int(i): 0 for i in range(o.M)}
        end = o.loads()
        add = {}
        for r in range(len(lens)):
            add[int(got["chosen"][r])] = add.get(int(got["chosen"][r]), 0) + int(lens[r]) - int(
                got["hit"][r][list(got["cand"][r]).index(got["chosen"][r])])
        for i in range(o.M):
            W[i] = int(end[i]) - add.get(i, 0)   # loads after the drain, before this batch's choices
        for r in range(len(lens)):
            c = [int(x) for x in got["cand"][r]]
            h = [int(x) for x in got["hit"][r]]
            L = int(lens[r])
            ttft = [W[c[f]] + (L - h[f]) for f in range(d)]
            assert [int(x) for x in got["ttft"][r]] == ttft
            top = max(h)
            tied = [f for f in range(d) if h[f] == top]
            a = min(tied, key=lambda f: (W[c[f]], f))
            pick = a
            over = len(tied) < d and ttft[a] > slo
            if over:
                pick = min(range(d), key=lambda f: (W[c[f]], 0 if f == a else 1, f))
            assert int(got["chosen"][r]) == c[pick], (bi, r)
            assert int(got["switched"][r]) == int(over)
            switched += pick != a
            W[c[pick]] += L - h[pick]
        o.commit()
    assert switched > 0


def test_identical_prompts_share_their_candidate_set():
    d, B = 4, 16
    o = mk(d, B=B)
    rng = np.random.default_rng(8)
    p = rng.integers(0, 1 << 32, size=20 * B, dtype=np.uint64).astype(np.uint32)
    n = 12
    tok = np.concatenate([p] * n)
    off = np.arange(n, dtype=np.uint64) * len(p)
    rc, out = o.route_batch_d(d, tok, off, np.full(n, len(p), np.uint32), 5)
    assert rc == 0
    assert all(out["cand"][r].tolist() == out["cand"][0].tolist() for r in range(n))
    # after a commit, every later copy hits on the instance that took the first
    o.commit()
    rc, out = o.route_batch_d(d, tok, off, np.full(n, len(p), np.uint32), 6)
    assert set(out["chosen"].tolist()) <= set(out["cand"][0].tolist())
    assert out["hit"].max() == len(p)


def test_two_choices_spread_load_more_than_one():
    """Distinct prompts, no cache reuse, an SLO of zero so the rule always
    falls back to the least loaded candidate: the busiest instance's request
    count drops sharply from d = 1 to d = 2 (App. A.8)."""
    B, n, M = 16, 4000, 16
    rng = np.random.default_rng(2)
    tok = rng.integers(0, 1 << 32, size=n * B, dtype=np.uint64).astype(np.uint32)
    off = np.arange(n, dtype=np.uint64) * B
    lens = np.full(n, B, np.uint32)
    peaks = {}
    for d in (1, 2, 3):
        o = mk(d, M=M, V=64, slo=0, B=B, K=1)
        rc, out = o.route_batch_d(d, tok, off, lens, 1)
        assert rc == 0
        peaks[d] = np.bincount(out["chosen"], minlength=M).max()
    assert peaks[1] - n / M > 4 * (peaks[2] - n / M)
    assert peaks[3] <= peaks[2] + 2


def test_d_candidate_argument_checks():
    o = mk(3, M=4, live=[0, 1, 2])
    tok = np.zeros(16, np.uint32)
    assert o.route_batch_d(4, tok, np.zeros(1, np.uint64), np.full(1, 16, np.uint32), 1)[0] == 1   # d > rings kept
    o2 = mk(4, M=5, live=[0, 1, 2])
    assert o2.route_batch_d(4, tok, np.zeros(1, np.uint64), np.full(1, 16, np.uint32), 1)[0] == 3  # d > live
    with pytest.raises(ValueError):
        mk(9)
