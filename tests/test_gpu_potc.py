"""The power-of-d-choices kernel (dm_potc_max_loads, App. A.8) against the
oracle: every trial's maximum load, bit for bit, over the paper's cluster
sizes and the edge cases (one bin, 256 bins, d = 64, trial counts that
leave a ragged last block)."""

import numpy as np
import pytest

from oracle import oracle as O
from parity_harness import lib_ready

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    lib_ready()


@pytest.mark.parametrize("n,m,d,trials", [(8, 8000, 1, 64), (8, 8000, 2, 100), (16, 16000, 2, 64),
                                          (24, 24000, 3, 33), (32, 32000, 4, 64), (1, 500, 2, 5),
                                          (256, 4000, 2, 70), (7, 3000, 64, 9), (32, 10, 2, 300),
                                          (4, 0, 2, 8)])
def test_potc_matches_oracle(n, m, d, trials):
    import torch
    from paper_2602_06502_gb300 import dualmap as D
    seed = 1000 + n * 7 + d
    out = torch.zeros(trials, dtype=torch.int32, device="cuda")
    assert D.dm_potc_max_loads(n, m, d, trials, seed, out) == 0
    torch.cuda.synchronize()
    got = out.cpu().numpy().astype(np.uint32)
    want = O.potc_max_loads(n, m, d, trials, seed)
    assert np.array_equal(got, want)


def test_potc_rejects_bad_arguments():
    import torch
    from paper_2602_06502_gb300 import dualmap as D
    out = torch.zeros(4, dtype=torch.int32, device="cuda")
    assert D.dm_potc_max_loads(0, 10, 2, 4, 1, out) == D.DM_ERR_INVALID_ARG
    assert D.dm_potc_max_loads(257, 10, 2, 4, 1, out) == D.DM_ERR_INVALID_ARG
    assert D.dm_potc_max_loads(8, 10, 65, 4, 1, out) == D.DM_ERR_INVALID_ARG
    assert D.dm_potc_max_loads(8, 1 << 32, 2, 4, 1, out) == D.DM_ERR_INVALID_ARG
    assert D.dm_potc_max_loads(8, 10, 2, 0, 1, out) == 0
