"""adapm_push_noalloc against adapm_push and the oracle, through the C ABI.

The allocation-free push serves callers that cannot let the library allocate
device memory during a call: a framework whose own allocator owns the device
memory budget, or a latency-critical loop in which cudaMalloc / cudaFree may
synchronise the device.  It runs the same kernels in the same summation order
as adapm_push, with its scratch in one file-scope device array shared by every
call, so its results must equal adapm_push's bit for bit, on calls in a row
whose scratch layouts shrink (leftovers of a larger earlier push, a longer
hot-key list or more chunks, must not leak into a smaller later one).  With
dyadic values every sum is exact in fp32, so the oracle's results are matched
bit for bit too.  This file runs last (its name), so that a failure here comes
after every other test has run.
"""
import numpy as np
import pytest
import torch

from oracle import ParameterManagerOracle

pytestmark = pytest.mark.gpu


def _pair(gpu_lib, K, D, W, init):
    a = gpu_lib.ParameterManager(K, D, W, init_values=torch.from_numpy(init).cuda())
    b = gpu_lib.ParameterManager(K, D, W, init_values=torch.from_numpy(init).cuda())
    return a, b


def _calls(rng, K, n_large):
    """Three pushes: a hot key over many chunks, two other hot keys, then a small cold one."""
    k1 = rng.integers(0, K, size=n_large)
    k1[rng.random(n_large) < 0.3] = 17
    k2 = rng.integers(0, K, size=n_large - 777)
    r = rng.random(k2.size)
    k2[r < 0.2] = 5
    k2[(r >= 0.2) & (r < 0.4)] = K - 1
    k3 = rng.integers(0, K, size=301)
    return [k1, k2, k3]


def _state(pm, K):
    allk = np.arange(K)
    val, acc, has = pm.replica_rows(1, allk)
    return pm.read_main(allk), val, acc, has


@pytest.mark.parametrize("K,D,n", [(5000, 64, 60000), (3000, 200, 20000)])
def test_push_noalloc_equals_push_bit_for_bit_on_calls_in_a_row(gpu_lib, K, D, n):
    W = 3
    rng = np.random.default_rng(D)
    init = rng.normal(0, 0.1, size=(K, D)).astype(np.float32)
    ref, noa = _pair(gpu_lib, K, D, W, init)
    # some keys get replicas of worker 1 so both kinds of target are exercised
    replicated = torch.as_tensor(rng.choice(K, size=K // 3, replace=False), device="cuda")
    for pm in (ref, noa):
        pm.intent(1, replicated, 0, 5)
    for call, keys in enumerate(_calls(rng, K, n)):
        keys_d = torch.as_tensor(keys, device="cuda")
        deltas = torch.from_numpy(rng.normal(0, 1e-3, size=(keys.size, D)).astype(np.float32)).cuda()
        ref.push(1, keys_d, deltas)
        noa.push_noalloc(1, keys_d, deltas)
        ref.wait()
        noa.wait()
        for x, y, name in zip(_state(ref, K), _state(noa, K), ("main", "value", "pending", "has")):
            assert np.array_equal(x, y), f"call {call}: {name} differs"
    assert ref.stats()["push_rows"] == noa.stats()["push_rows"]
    ref.close()
    noa.close()


def test_push_noalloc_dyadic_matches_oracle(gpu_lib):
    K, D, W = 4000, 64, 2
    rng = np.random.default_rng(7)
    init = (rng.integers(-1024, 1025, size=(K, D)) * 2.0 ** -10).astype(np.float32)
    pm = gpu_lib.ParameterManager(K, D, W, init_values=torch.from_numpy(init).cuda())
    ref = ParameterManagerOracle(K, D, W, init)
    rep = rng.choice(K, size=K // 4, replace=False)
    pm.intent(1, torch.as_tensor(rep, device="cuda"), 0, 3)
    ref.intent(1, rep, 0, 3)
    for call, keys in enumerate(_calls(rng, K, 50000)):
        d = (rng.integers(-64, 65, size=(keys.size, D)) * 2.0 ** -10).astype(np.float32)
        pm.push_noalloc(1, torch.as_tensor(keys, device="cuda"), torch.from_numpy(d).cuda())
        ref.push(1, keys, d)
        pm.wait()
        allk = np.arange(K)
        assert np.array_equal(pm.read_main(allk), ref.read_main(allk)), f"call {call}: main"
        ks, val, acc = ref.replica_values(1)
        gval, gacc, has = pm.replica_rows(1, ks)
        assert has.all() and np.array_equal(gval, val) and np.array_equal(gacc, acc), f"call {call}: replicas"
    pm.close()


def test_push_noalloc_rejects_what_it_cannot_serve(gpu_lib):
    A = gpu_lib
    K, D = 100, 64
    pm = A.ParameterManager(K, D, 1)
    # host arrays would need staging buffers
    with pytest.raises(A.AdaPMError) as e:
        pm.push_noalloc(0, np.array([1, 2]), np.zeros((2, D), np.float32))
    assert e.value.status == A.EINVAL
    # more rows than the 16 MiB scratch holds (about 790k at value_len 64)
    n = 900000
    with pytest.raises(A.AdaPMError) as e:
        pm.push_noalloc(0, torch.zeros(n, dtype=torch.int32, device="cuda"),
                        torch.zeros((n, D), device="cuda"))
    assert e.value.status == A.EINVAL and "scratch" in str(e.value)
    assert "scratch" in pm.last_error()
    # nothing was applied, the context still works, and a call that succeeds clears the message
    pm.push_noalloc(0, torch.tensor([3], device="cuda"), torch.ones((1, D), device="cuda"))
    assert pm.last_error() == ""
    pm.wait()
    assert np.array_equal(pm.read_main([3]), np.ones((1, D), np.float32))
    assert not pm.read_main([0]).any()
    pm.close()


def test_push_noalloc_is_profiled_like_push(gpu_lib):
    K, D = 1000, 64
    pm = gpu_lib.ParameterManager(K, D, 1)
    pm.profile_enable(True)
    pm.profile_read()
    keys = torch.randint(0, K, (5000,), device="cuda")
    pm.push_noalloc(0, keys, torch.ones((5000, D), device="cuda"))
    prof = pm.profile_read()
    assert prof["push"][1] == 1 and prof["push_kernel"][1] == 1
    assert prof["push"][0] >= prof["push_kernel"][0] > 0
    pm.close()
