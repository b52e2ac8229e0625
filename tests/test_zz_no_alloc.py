"""adapm_push_noalloc against adapm_push, through the C ABI.

The allocation-free push is for callers that cannot let the library allocate
device memory during a call (a framework whose allocator owns the memory
budget, or a latency-critical loop where cudaMalloc/cudaFree may synchronise
the device).  It must give the same result as the ordinary push.  Two calls
in a row check that the shared scratch array's leftover contents from the
first call do not leak into the second.  Runs last (file name) so that a
failure here comes after every other test has run.
"""
import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu

RTOL = 1e-5


def _pair(gpu_lib, K, D, W, init):
    a = gpu_lib.ParameterManager(K, D, W, init_values=torch.from_numpy(init).cuda())
    b = gpu_lib.ParameterManager(K, D, W, init_values=torch.from_numpy(init).cuda())
    return a, b


@pytest.mark.parametrize("K,D,n", [(5000, 64, 60000), (3000, 200, 20000)])
def test_push_noalloc_matches_push_on_two_calls(gpu_lib, K, D, n):
    W = 3
    rng = np.random.default_rng(D)
    init = rng.normal(0, 0.1, size=(K, D)).astype(np.float32)
    ref, noa = _pair(gpu_lib, K, D, W, init)
    # some keys get replicas of worker 1 so both kinds of target are exercised
    replicated = torch.as_tensor(rng.choice(K, size=K // 3, replace=False), device="cuda")
    for pm in (ref, noa):
        pm.intent(1, replicated, 0, 5)
    for call in range(2):
        keys = rng.integers(0, K, size=n)
        keys[rng.random(n) < 0.3] = 17                     # a hot key spanning many chunks
        keys_d = torch.as_tensor(keys, device="cuda")
        deltas = torch.from_numpy(rng.normal(0, 1e-3, size=(n, D)).astype(np.float32)).cuda()
        ref.push(1, keys_d, deltas)
        noa.push_noalloc(1, keys_d, deltas)
        ref.wait()
        noa.wait()
        allk = np.arange(K)
        m_ref, m_noa = ref.read_main(allk), noa.read_main(allk)
        v_ref, a_ref, h_ref = ref.replica_rows(1, allk)
        v_noa, a_noa, h_noa = noa.replica_rows(1, allk)
        assert np.array_equal(h_ref, h_noa)
        for x, y in ((m_ref, m_noa), (v_ref, v_noa), (a_ref, a_noa)):
            assert np.all(np.abs(x - y) <= RTOL * np.abs(x) + 1e-7), f"call {call}"
    ref.close()
    noa.close()


def test_push_noalloc_rejects_what_it_cannot_serve(gpu_lib):
    A = gpu_lib
    K, D = 100, 1024
    pm = A.ParameterManager(K, D, 1)
    # host arrays would need staging buffers
    with pytest.raises(A.AdaPMError) as e:
        pm.push_noalloc(0, np.array([1, 2]), np.zeros((2, D), np.float32))
    assert e.value.status == A.EINVAL
    # more rows than the 16 MiB scratch holds at value_len 1024
    n = 40000
    with pytest.raises(A.AdaPMError) as e:
        pm.push_noalloc(0, torch.zeros(n, dtype=torch.int32, device="cuda"),
                        torch.zeros((n, D), device="cuda"))
    assert e.value.status == A.EINVAL and "scratch" in str(e.value)
    # nothing was applied, and the context still works
    pm.push_noalloc(0, torch.tensor([3], device="cuda"), torch.ones((1, D), device="cuda"))
    pm.wait()
    assert np.array_equal(pm.read_main([3]), np.ones((1, D), np.float32))
    assert not pm.read_main([0]).any()
    pm.close()
