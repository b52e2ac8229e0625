"""adapm_pull with rows staged in shared memory by the bulk-copy engine (pull_staging) against the
register gather and the oracle: pulled rows are copies, so they must be equal bit for bit, for
replicated and main-copy rows, repeated keys, a ragged last tile, keys out of range (zero rows,
ERANGE) and row widths from 16 bytes to 4 KB (the tile shrinks as rows grow)."""
import numpy as np
import pytest
import torch

from oracle import ParameterManagerOracle
from tests.seqgen import dyadic_init

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("K,D,n", [(3000, 4, 1000), (50000, 64, 300001), (4000, 200, 7777), (800, 1024, 333)])
def test_bulk_pull_equals_register_pull_and_oracle(gpu_lib, K, D, n):
    W = 2
    rng = np.random.default_rng(D)
    init = dyadic_init(K, D, 1)
    pms = [gpu_lib.ParameterManager(K, D, W, init_values=torch.from_numpy(init).cuda(), pull_staging=st)
           for st in (False, True)]
    ref = ParameterManagerOracle(K, D, W, init)
    rep = rng.choice(K, size=K // 2, replace=False)
    for pm in pms:
        pm.intent(1, torch.as_tensor(rep, device="cuda"), 0, 3)
    ref.intent(1, rep, 0, 3)
    # replica values that differ from main, so the source of every row shows
    d = (rng.integers(-64, 65, size=(rep.size, D)) * 2.0 ** -10).astype(np.float32)
    for pm in pms:
        pm.push(1, torch.as_tensor(rep, device="cuda"), torch.from_numpy(d).cuda())
    ref.push(1, rep, d)
    keys = rng.integers(0, K, size=n)
    for w in range(W):
        outs = [pm.pull(w, torch.as_tensor(keys, device="cuda")) for pm in pms]
        for pm in pms:
            pm.wait()
        a, b = (o.cpu().numpy() for o in outs)
        assert np.array_equal(a, b)
        assert np.array_equal(b, ref.pull(w, keys))
    # keys out of range: zero rows and ERANGE, the same on both paths
    bad = keys[:97].copy()
    bad[[0, 50, 96]] = K + 7
    for pm in pms:
        out = pm.pull(1, torch.as_tensor(bad, device="cuda"))
        with pytest.raises(gpu_lib.AdaPMError) as e:
            pm.wait()
        assert e.value.status == gpu_lib.ERANGE
        got = out.cpu().numpy()
        assert not got[[0, 50, 96]].any()
        good = np.setdiff1d(np.arange(97), [0, 50, 96])
        assert np.array_equal(got[good], ref.pull(1, bad[good]))
    for pm in pms:
        pm.close()
