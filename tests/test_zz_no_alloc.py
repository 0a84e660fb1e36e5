"""dm_hash_prompts_noalloc: the hashing entry point for callers that cannot
allocate device memory (its working memory is a fixed array inside the
library) must return exactly what dm_hash_prompts returns on a handle with the
same block size, route-prefix length and seed, call after call (the array is
shared and keeps the previous call's contents), and refuse sizes beyond its
stated limits.  This file is collected last on purpose."""

import ctypes as C

import numpy as np
import pytest

from parity_harness import lib_ready

pytestmark = pytest.mark.gpu


def _batch(rng, B, n, maxlen):
    lens = rng.integers(B, maxlen, size=n).astype(np.uint32)
    lens[0] = B                       # edge lengths: one block, one block + 1
    lens[1] = B + 1
    off = np.zeros(n, np.uint64)
    off[1:] = np.cumsum((lens[:-1].astype(np.uint64) + 3) // 4 * 4)
    ntok = int(off[-1] + lens[-1])
    tok = rng.integers(0, 1 << 32, size=ntok + 4, dtype=np.uint64).astype(np.uint32)
    return tok, off, lens, ntok


def _run(fn, torch, D, tok, off, lens, ntok):
    dt = torch.from_numpy(tok.view(np.int32)).cuda()
    do = torch.from_numpy(off.view(np.int64)).cuda()
    dl = torch.from_numpy(lens.view(np.int32)).cuda()
    nkeys = int((lens // fn.B).sum())
    keys = torch.full((nkeys + 1,), -1, dtype=torch.int64, device="cuda")
    koff = torch.full((len(lens) + 1,), -1, dtype=torch.int64, device="cuda")
    pos = torch.full((2 * len(lens),), -1, dtype=torch.int64, device="cuda")
    b = D.make_batch(dt, do, dl, len(lens), ntok, 0)
    rc = fn(b, keys, koff, pos)
    torch.cuda.synchronize()
    return rc, keys[:nkeys].cpu().numpy(), koff.cpu().numpy(), pos.cpu().numpy()


@pytest.mark.parametrize("B,K", [(16, 16), (8, 40)])
def test_noalloc_matches_dm_hash_prompts_twice(B, K):
    lib_ready()
    import torch
    from paper_2602_06502_gb300 import dualmap as D
    from paper_2602_06502_gb300.scheduler import Scheduler
    seed = 4242 + B
    g = Scheduler(block_tokens=B, route_prefix_blocks=K, vnodes=4, max_instances=4, capacity=16, max_batch=512,
                  max_batch_tokens=1 << 24, seed=seed)
    stream = C.c_void_p(torch.cuda.current_stream().cuda_stream)

    def ref(b, keys, koff, pos):
        rc = D.dm_hash_prompts(g.h, b, keys, koff, pos)
        return rc or g.last_error()

    def noalloc(b, keys, koff, pos):
        return D.dm_hash_prompts_noalloc(B, K, seed, b, keys, koff, pos, stream)

    ref.B = noalloc.B = B
    rng = np.random.default_rng(B * 7 + K)
    # two calls in a row with different batches: the shared array must not
    # leak the first call's contents into the second
    for n, maxlen in ((300, 40 * B * 64), (37, 3 * B * 64)):
        tok, off, lens, ntok = _batch(rng, B, n, maxlen)
        want = _run(ref, torch, D, tok, off, lens, ntok)
        got = _run(noalloc, torch, D, tok, off, lens, ntok)
        assert want[0] == 0 and got[0] == 0
        for w, x in zip(want[1:], got[1:]):
            assert np.array_equal(w, x)
    g.close()


def test_noalloc_matches_the_oracle():
    """The same keys and positions as the CPU oracle, prompt by prompt (no
    handle involved at all)."""
    lib_ready()
    import torch
    from oracle import oracle as O
    from paper_2602_06502_gb300 import dualmap as D
    B, K, seed = 16, 16, 777
    stream = C.c_void_p(torch.cuda.current_stream().cuda_stream)
    ora = O.Oracle(block_tokens=B, route_prefix_blocks=K, vnodes_per_instance=4, max_instances=4,
                   cache_capacity_blocks=16, slo_us=1, cost_us_per_token=1, hot_num=3, hot_den=2,
                   max_batch=64, max_batch_tokens=1 << 22, seed=seed)

    def noalloc(b, keys, koff, pos):
        return D.dm_hash_prompts_noalloc(B, K, seed, b, keys, koff, pos, stream)

    noalloc.B = B
    tok, off, lens, ntok = _batch(np.random.default_rng(5), B, 40, 9 * B * 64)
    rc, keys, koff, pos = _run(noalloc, torch, D, tok, off, lens, ntok)
    assert rc == 0
    for r in range(len(lens)):
        want_k, want_p = ora.prompt_keys(tok[int(off[r]):int(off[r]) + int(lens[r])])
        assert np.array_equal(keys[int(koff[r]):int(koff[r + 1])].view(np.uint64), want_k), r
        assert np.array_equal(pos[2 * r:2 * r + 2].view(np.uint64), want_p), r


def test_noalloc_reports_device_side_errors_and_recovers():
    """Errors only the device can see come back from the call itself, and
    the next valid call is unaffected: a prompt shorter than a block
    (DM_ERR_INVALID_ARG), and prompts that overlap so much that their exact
    block count passes DM_NOALLOC_MAX_BLOCKS while total_tokens / B stays
    within it (DM_ERR_CAPACITY)."""
    lib_ready()
    import torch
    from paper_2602_06502_gb300 import dualmap as D
    from paper_2602_06502_gb300.scheduler import Scheduler
    B, K, seed = 16, 16, 99
    stream = C.c_void_p(torch.cuda.current_stream().cuda_stream)

    def noalloc(b, keys, koff, pos):
        return D.dm_hash_prompts_noalloc(B, K, seed, b, keys, koff, pos, stream)

    noalloc.B = B
    rng = np.random.default_rng(11)
    tok, off, lens, ntok = _batch(rng, B, 8, 4 * B * 64)
    short = lens.copy()
    short[3] = B - 1
    assert _run(noalloc, torch, D, tok, off, short, ntok)[0] == D.DM_ERR_INVALID_ARG
    # two prompts over the same 3,000,000 blocks: 6,000,000 keyed blocks in a
    # buffer of 3,000,000 blocks (DM_NOALLOC_MAX_BLOCKS = 4,194,304)
    nb_each = 3_000_000
    big_tok = torch.zeros(nb_each * B + 4, dtype=torch.int32, device="cuda")
    dofs = torch.zeros(2, dtype=torch.int64, device="cuda")
    dlen = torch.full((2,), nb_each * B, dtype=torch.int32, device="cuda")
    keys = torch.zeros(2 * nb_each + 1, dtype=torch.int64, device="cuda")
    koff = torch.zeros(3, dtype=torch.int64, device="cuda")
    pos = torch.zeros(4, dtype=torch.int64, device="cuda")
    b = D.make_batch(big_tok, dofs, dlen, 2, nb_each * B, 0)
    assert D.dm_hash_prompts_noalloc(B, K, seed, b, keys, koff, pos, stream) == D.DM_ERR_CAPACITY
    del big_tok, keys
    # the next valid call matches dm_hash_prompts
    g = Scheduler(block_tokens=B, route_prefix_blocks=K, vnodes=4, max_instances=4, capacity=16, max_batch=64,
                  max_batch_tokens=1 << 22, seed=seed)

    def ref(b, keys, koff, pos):
        rc = D.dm_hash_prompts(g.h, b, keys, koff, pos)
        return rc or g.last_error()

    ref.B = B
    want = _run(ref, torch, D, tok, off, lens, ntok)
    got = _run(noalloc, torch, D, tok, off, lens, ntok)
    assert want[0] == 0 and got[0] == 0
    for w, x in zip(want[1:], got[1:]):
        assert np.array_equal(w, x)
    g.close()


def test_noalloc_rejects_sizes_beyond_its_limits():
    lib_ready()
    import torch
    from paper_2602_06502_gb300 import dualmap as D
    stream = C.c_void_p(torch.cuda.current_stream().cuda_stream)
    dummy = torch.zeros(16, dtype=torch.int64, device="cuda")
    n_over = 4097                                   # DM_NOALLOC_MAX_REQUESTS + 1
    b = D.make_batch(dummy, dummy, dummy, n_over, 64, 0)
    assert D.dm_hash_prompts_noalloc(16, 16, 1, b, dummy, dummy, dummy, stream) == D.DM_ERR_CAPACITY
    b = D.make_batch(dummy, dummy, dummy, 1, 16 * 4194304 + 16, 0)   # more than DM_NOALLOC_MAX_BLOCKS
    assert D.dm_hash_prompts_noalloc(16, 16, 1, b, dummy, dummy, dummy, stream) == D.DM_ERR_CAPACITY
