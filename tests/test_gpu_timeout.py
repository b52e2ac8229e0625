"""The bounded grid-barrier wait of the push's key sort, made to run out.

No GPU fault is involved: adapm_debug_fail_next_barrier makes the next
push's sort wait for barrier arrivals that never come.  The wait gives up
after about a second, the kernels that consume the sort leave the store
untouched, adapm_wait reports ADAPM_ETIMEOUT and retires the context, and a
new context on the same GPU works normally.
"""
import time

import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu


def test_barrier_wait_gives_up_and_leaves_the_store(gpu_lib):
    A = gpu_lib
    K, D, W = 1000, 8, 1
    init = (np.arange(K * D, dtype=np.float32).reshape(K, D) * 2.0 ** -4)
    pm = A.ParameterManager(K, D, W, init_values=torch.from_numpy(init).cuda())
    keys = torch.arange(0, 100, device="cuda", dtype=torch.int32)
    deltas = torch.ones(100, D, device="cuda")
    pm.push(0, keys, deltas)
    pm.wait()
    before = pm.read_main(np.arange(K))
    assert np.array_equal(before[:100], init[:100] + 1)
    pm.debug_fail_next_barrier()
    t0 = time.time()
    pm.push(0, keys, deltas)
    after = pm.read_main(np.arange(K))   # synchronises with the failed push
    elapsed = time.time() - t0
    assert np.array_equal(after, before), "a push whose sort gave up must not touch the store"
    assert elapsed < 60.0
    with pytest.raises(A.AdaPMError) as e:
        pm.wait()
    assert e.value.status == A.ETIMEOUT
    with pytest.raises(A.AdaPMError) as e:
        pm.push(0, keys, deltas)
    assert e.value.status == A.ECUDA   # the context is retired
    pm.close()
    # the GPU and new contexts are unaffected
    pm2 = A.ParameterManager(K, D, W, init_values=torch.from_numpy(init).cuda())
    pm2.push(0, keys, deltas)
    pm2.wait()
    assert np.array_equal(pm2.read_main(np.arange(K)), before)
    pm2.close()


@pytest.mark.parametrize("call", ["push", "push_noalloc", "pull"])
def test_launch_failure_retires_the_context(gpu_lib, call):
    """A CUDA error after a call's launches (injected on the host: no GPU fault) retires the context, for the
    allocation-free push as for every other entry point; later calls report it and other contexts work."""
    A = gpu_lib
    K, D = 500, 8
    pm = A.ParameterManager(K, D, 1)
    keys = torch.arange(0, 64, device="cuda", dtype=torch.int32)
    deltas = torch.ones(64, D, device="cuda")
    pm.push(0, keys, deltas)
    pm.wait()
    pm.debug_fail_next_launch()
    with pytest.raises(A.AdaPMError) as e:
        if call == "pull":
            pm.pull(0, keys)
        else:
            getattr(pm, call)(0, keys, deltas)
    assert e.value.status == A.ECUDA
    assert pm.last_error() != ""
    for retry in (lambda: pm.push(0, keys, deltas), lambda: pm.push_noalloc(0, keys, deltas), pm.wait):
        with pytest.raises(A.AdaPMError) as e:
            retry()
        assert e.value.status == A.ECUDA
    pm.close()
    pm2 = A.ParameterManager(K, D, 1)
    pm2.push_noalloc(0, keys, deltas)
    pm2.wait()
    assert np.array_equal(pm2.read_main(np.arange(64)), np.ones((64, D), np.float32))
    pm2.close()
