"""Pins of the oracle's hashing: published test vectors for its primitives,
closed forms for NH, the digest chain and the cache-key mapping, and the
prefix-locality property the paper relies on (a key identifies its prefix)."""

import json
import os

import numpy as np
import pytest

from oracle import oracle as O

GOLD = os.path.join(os.path.dirname(__file__), "golden")
M64 = (1 << 64) - 1
M32 = (1 << 32) - 1


def _gold(name):
    with open(os.path.join(GOLD, name)) as f:
        return json.load(f)


def test_splitmix64_published_vector():
    g = _gold("published_vectors.json")["splitmix64_seed_1234567_first5"]
    assert O.splitmix64_stream(1234567, 5) == g["values"]


def test_mix64_is_one_splitmix_step():
    for x in (0, 1, 1234567, M64, 0x0123456789ABCDEF):
        assert O.mix64(x) == O.splitmix64_stream(x, 1)[0]


def _murmur3_x64_128(data, seed, fmix):
    """MurmurHash3_x64_128 body (Appleby) with the finaliser supplied."""
    def rotl(x, r):
        return ((x << r) | (x >> (64 - r))) & M64
    c1, c2 = 0x87C37B91114253D5, 0x4CF5AD432745937F
    h1 = h2 = seed
    n = len(data)
    nb = n // 16
    for i in range(nb):
        k1 = int.from_bytes(data[16 * i:16 * i + 8], "little")
        k2 = int.from_bytes(data[16 * i + 8:16 * i + 16], "little")
        k1 = rotl((k1 * c1) & M64, 31) * c2 & M64
        h1 ^= k1
        h1 = (rotl(h1, 27) + h2) & M64
        h1 = (h1 * 5 + 0x52DCE729) & M64
        k2 = rotl((k2 * c2) & M64, 33) * c1 & M64
        h2 ^= k2
        h2 = (rotl(h2, 31) + h1) & M64
        h2 = (h2 * 5 + 0x38495AB5) & M64
    tail = data[16 * nb:]
    k1 = k2 = 0
    for i in range(len(tail) - 1, 7, -1):
        k2 ^= tail[i] << (8 * (i - 8))
    if len(tail) > 8:
        h2 ^= rotl((k2 * c2) & M64, 33) * c1 & M64
    for i in range(min(len(tail), 8) - 1, -1, -1):
        k1 ^= tail[i] << (8 * i)
    if len(tail) > 0:
        h1 ^= rotl((k1 * c1) & M64, 31) * c2 & M64
    h1 ^= n
    h2 ^= n
    h1 = (h1 + h2) & M64
    h2 = (h2 + h1) & M64
    h1, h2 = fmix(h1), fmix(h2)
    h1 = (h1 + h2) & M64
    h2 = (h2 + h1) & M64
    return h1.to_bytes(8, "little") + h2.to_bytes(8, "little")


def test_fmix64_via_smhasher_verification_value():
    """The oracle's fmix64 inside MurmurHash3_x64_128 reproduces SMHasher's
    published verification value; any wrong constant or shift breaks it."""
    g = _gold("published_vectors.json")["murmurhash3_x64_128_verification"]
    key = bytearray()
    digests = bytearray()
    for i in range(256):
        digests += _murmur3_x64_128(bytes(key), 256 - i, O.fmix64)
        key.append(i)
    final = _murmur3_x64_128(bytes(digests), 0, O.fmix64)
    assert int.from_bytes(final[:4], "little") == g["value"]


def _fmix64_inverse(y):
    """Inverse of the MurmurHash3 finaliser (xorshift-33 is an involution;
    the multipliers are odd, so invertible mod 2^64)."""
    y ^= y >> 33
    y = (y * pow(0xC4CEB9FE1A85EC53, -1, 1 << 64)) & M64
    y ^= y >> 33
    y = (y * pow(0xFF51AFD7ED558CCD, -1, 1 << 64)) & M64
    y ^= y >> 33
    return y


def test_fmix64_inverse_roundtrip():
    rng = np.random.default_rng(7)
    for x in rng.integers(0, 2**63, size=50, dtype=np.int64).tolist() + [0, 1, M64]:
        assert _fmix64_inverse(O.fmix64(x)) == x


# -- NH (UMAC) closed forms -------------------------------------------------

@pytest.mark.parametrize("B", [4, 8, 16, 32, 64])
def test_nh_cancelling_tokens_give_zero(B):
    rng = np.random.default_rng(B)
    K = rng.integers(0, 2**32, size=B, dtype=np.uint64).astype(np.uint32)
    t = ((1 << 32) - K.astype(np.uint64)).astype(np.uint64) & M32
    assert O.nh(t.astype(np.uint32), K) == 0


@pytest.mark.parametrize("B", [4, 16, 64])
def test_nh_single_pair(B):
    """Only pair i survives the keying: NH equals that one product, for
    every i (catches a mis-paired or shifted index)."""
    rng = np.random.default_rng(100 + B)
    K = rng.integers(0, 2**32, size=B, dtype=np.uint64)
    for i in range(B // 2):
        a, b = int(rng.integers(1, 2**32)), int(rng.integers(1, 2**32))
        t = (-K) & M32
        t[2 * i] = (a - int(K[2 * i])) & M32
        t[2 * i + 1] = (b - int(K[2 * i + 1])) & M32
        assert O.nh(t.astype(np.uint32), K.astype(np.uint32)) == (a * b) & M64


def test_nh_wraps_mod_2_64():
    B = 16
    K = np.zeros(B, np.uint32)
    t = np.full(B, M32, np.uint32)
    assert O.nh(t, K) == ((B // 2) * M32 * M32) & M64


def test_nh_zero_tokens_is_key_products():
    B = 16
    K = np.arange(1, B + 1, dtype=np.uint32) * np.uint32(0x10001)
    t = np.zeros(B, np.uint32)
    want = sum(int(K[2 * i]) * int(K[2 * i + 1]) for i in range(B // 2)) & M64
    assert O.nh(t, K) == want


# -- key material ---------------------------------------------------------

def test_key_material_draw_order():
    seed, B = 99, 16
    draws = O.splitmix64_stream(seed, 2 * B + 7)
    K1, K2, sc = O.derive_keys(seed, B)
    assert K1.tolist() == [d & M32 for d in draws[:B]]
    assert K2.tolist() == [d & M32 for d in draws[B:2 * B]]
    assert int(sc[0]) == draws[2 * B] | 1 and int(sc[1]) == draws[2 * B + 1] | 1
    assert [int(x) for x in sc[2:]] == draws[2 * B + 2:2 * B + 7]


# -- the chain, cache keys and route positions -------------------------------

def _oracle(B=16, K=16, seed=5):
    return O.Oracle(block_tokens=B, route_prefix_blocks=K, vnodes_per_instance=4, max_instances=8,
                    cache_capacity_blocks=1024, slo_us=10**6, cost_us_per_token=1, hot_num=3,
                    hot_den=2, max_batch=64, max_batch_tokens=1 << 24, seed=seed)


def _cancel(K, nblk, B):
    return np.tile(((1 << 32) - K.astype(np.uint64)) & M32, nblk).astype(np.uint32)


@pytest.mark.parametrize("B,Kr", [(16, 16), (4, 3), (64, 2)])
def test_chain_closed_form_zero_nh(B, Kr):
    """With NH cancelled in every block, d_k = fmix64((k+1) G1), so
    P_b = sum_{k<=b} fmix64((k+1) G1) and key_b = fmix64(P_b ^ S_c)."""
    o = _oracle(B, Kr)
    K1, K2, sc = o.key_material()
    G1, Sc, Sr1 = int(sc[0]), int(sc[2]), int(sc[3])
    nblk = 21
    tok = _cancel(K1, nblk, B)
    tok = np.concatenate([tok, np.arange(B - 1, dtype=np.uint32)])  # partial tail, never keyed
    keys, pos = o.prompt_keys(tok)
    assert len(keys) == nblk
    P = 0
    for b in range(nblk):
        P = (P + O.fmix64(((b + 1) * G1) & M64)) & M64
        k = O.fmix64(P ^ Sc)
        assert int(keys[b]) == (k if k else 1)
        if b == min(Kr, nblk) - 1:
            assert int(pos[0]) == O.fmix64(P ^ Sr1)


def test_route_position_two_closed_form():
    """Second function: cancel NH under K2; pos2 = fmix64(sum_{k<K} fmix64((k+1) G2) ^ S_r2)."""
    B, Kr = 16, 5
    o = _oracle(B, Kr)
    K1, K2, sc = o.key_material()
    G2, Sr2 = int(sc[1]), int(sc[4])
    for nblk in (3, 5, 9):      # fewer blocks than K_route uses all of them
        _, pos = o.prompt_keys(_cancel(K2, nblk, B))
        P = 0
        for k in range(min(Kr, nblk)):
            P = (P + O.fmix64(((k + 1) * G2) & M64)) & M64
        assert int(pos[1]) == O.fmix64(P ^ Sr2)


def test_cache_key_zero_maps_to_one():
    """Build block 0 so that P_0 == S_c, making fmix64(P_0 ^ S_c) == 0."""
    B = 16
    o = _oracle(B)
    K1, _, sc = o.key_material()
    G1, Sc = int(sc[0]), int(sc[2])
    target = (_fmix64_inverse(Sc) - G1) & M64     # nh_0 must equal this
    a, c = target >> 32, target & M32
    # target = a*(2^32-1) + a*1 + c*1 using three NH pairs
    vals = [(a, M32), (a, 1), (c, 1)] + [(0, 0)] * (B // 2 - 3)
    t = np.zeros(B, np.uint64)
    for i, (x, y) in enumerate(vals):
        t[2 * i] = (x - int(K1[2 * i])) & M32
        t[2 * i + 1] = (y - int(K1[2 * i + 1])) & M32
    assert O.nh(t.astype(np.uint32), K1) == target
    keys, _ = o.prompt_keys(t.astype(np.uint32))
    assert int(keys[0]) == 1


def test_prefix_locality():
    """Changing block j leaves keys of blocks < j unchanged and changes every
    key >= j (the key of block b identifies the whole prefix 0..b)."""
    B = 16
    o = _oracle(B)
    rng = np.random.default_rng(3)
    tok = rng.integers(0, 32000, size=B * 40 + 7, dtype=np.uint32)
    k0, p0 = o.prompt_keys(tok)
    for j in (0, 1, 15, 16, 39):
        t2 = tok.copy()
        t2[j * B + 3] ^= 1
        k1, p1 = o.prompt_keys(t2)
        assert np.array_equal(k0[:j], k1[:j])
        assert np.all(k0[j:] != k1[j:])
        assert (p0[0] != p1[0]) == (j < 16) and (p0[1] != p1[1]) == (j < 16)
    t3 = tok.copy()
    t3[-1] ^= 5                    # tail token: no effect at all
    k3, p3 = o.prompt_keys(t3)
    assert np.array_equal(k0, k3) and np.array_equal(p0, p3)


def test_route_prefix_shared_only():
    """Prompts equal on the first K_route blocks share both positions."""
    B, Kr = 16, 16
    o = _oracle(B, Kr)
    rng = np.random.default_rng(4)
    pre = rng.integers(0, 32000, size=B * Kr, dtype=np.uint32)
    a = np.concatenate([pre, rng.integers(0, 32000, size=333, dtype=np.uint32)])
    b = np.concatenate([pre, rng.integers(0, 32000, size=1000, dtype=np.uint32)])
    _, pa = o.prompt_keys(a)
    _, pb = o.prompt_keys(b)
    assert np.array_equal(pa, pb)
    ka, _ = o.prompt_keys(a)
    kb, _ = o.prompt_keys(b)
    assert np.array_equal(ka[:Kr], kb[:Kr]) and ka[Kr] != kb[Kr]


def test_block_shift_changes_digest():
    """The same block content at another index gives another digest: the
    salt (k+1) G enters each digest (a permuted prompt keys differently)."""
    B = 16
    o = _oracle(B)
    rng = np.random.default_rng(9)
    x = rng.integers(0, 32000, size=B, dtype=np.uint32)
    y = rng.integers(0, 32000, size=B, dtype=np.uint32)
    kxy, _ = o.prompt_keys(np.concatenate([x, y]))
    kyx, _ = o.prompt_keys(np.concatenate([y, x]))
    assert kxy[1] != kyx[1]


def test_key_uniformity():
    """Avalanche sanity: top-bit and bucket occupancy of random keys."""
    o = _oracle(16)
    rng = np.random.default_rng(11)
    keys = np.concatenate([o.prompt_keys(rng.integers(0, 32000, size=16 * 64, dtype=np.uint32))[0]
                           for _ in range(64)])
    top = (keys >> np.uint64(63)).astype(np.int64)
    assert abs(top.mean() - 0.5) < 0.05
    hist = np.bincount((keys & np.uint64(15)).astype(np.int64), minlength=16)
    assert hist.min() > 0.5 * hist.mean()
