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
