"""GPU parity of the versioned refresh (App. B.1.2: holders receive only updates they have not seen).

With delta_refresh the sync leaves a sole holder's value alone when nobody else wrote the key since its last
sync.  The CUDA path and the oracle run the same seeded call sequences: bit-exact with dyadic deltas (replica
sets, pulls, every stored value) and the same number of refreshed replicas, with and without relocation; the
hand-built case in which the holder's own fp32 rounding and main's differ; gaussian deltas within 1e-5 of the
magnitude bound.
"""
import numpy as np
import pytest
import torch

from oracle import ParameterManagerOracle
from tests.seqgen import dyadic_init, random_sequence
from tests.test_gpu_store import RTOL, apply_gpu, apply_ref, compare_full_state, dev

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("relocate", [False, True])
@pytest.mark.parametrize("K,D,W,max_batch,n_ops", [(40, 4, 3, 12, 300), (3000, 64, 4, 4000, 60),
                                                   (900, 200, 2, 2500, 40)])
def test_random_sequences_versioned_refresh_bit_exact(gpu_lib, relocate, K, D, W, max_batch, n_ops):
    init = dyadic_init(K, D, 8)
    pm = gpu_lib.ParameterManager(K, D, W, init_values=torch.from_numpy(init).cuda(), relocate=relocate,
                                  delta_refresh=True)
    ref = ParameterManagerOracle(K, D, W, init, relocation=relocate, delta_refresh=True)
    for i, op in enumerate(random_sequence(K * 3 + W, K, D, W, n_ops, max_batch=max_batch)):
        got = apply_gpu(pm, op)
        want = apply_ref(ref, op)
        if op["op"] == "pull":
            assert np.array_equal(got, want), f"pull {i}"
    compare_full_state(pm, ref, K, W)
    pm.sync()
    ref.sync()
    compare_full_state(pm, ref, K, W)
    assert pm.stats()["sync_refreshed"] == ref.refreshed
    pm.close()


def test_sole_holder_keeps_its_own_rounding_on_gpu(gpu_lib):
    for delta_refresh, want_val in ((True, 1.0), (False, 1.0 + 2.0 ** -23)):
        pm = gpu_lib.ParameterManager(1, 4, 1, init_values=torch.ones(1, 4, device="cuda"),
                                      delta_refresh=delta_refresh)
        pm.intent(0, dev([0]), 0, 9)
        for _ in range(2):
            pm.push(0, dev([0]), torch.full((1, 4), 2.0 ** -24, device="cuda"))
        pm.sync()
        pm.wait()
        assert pm.read_main(np.array([0]))[0, 0] == np.float32(1.0 + 2.0 ** -23)
        assert pm.pull(0, dev([0])).cpu().numpy()[0, 0] == np.float32(want_val)
        assert pm.stats()["sync_refreshed"] == (0 if delta_refresh else 1)
        pm.close()


def test_versioned_refresh_gaussian_within_tolerance(gpu_lib):
    K, D, W = 2000, 64, 4
    rng = np.random.default_rng(5)
    init = rng.normal(0, 0.1, size=(K, D)).astype(np.float32)
    pm = gpu_lib.ParameterManager(K, D, W, init_values=torch.from_numpy(init).cuda(), delta_refresh=True)
    ref = ParameterManagerOracle(K, D, W, init, delta_refresh=True)
    mag = ParameterManagerOracle(K, D, W, np.abs(init), delta_refresh=True)
    for op in random_sequence(606, K, D, W, 80, max_batch=3000, gaussian=True):
        got = apply_gpu(pm, op)
        want = apply_ref(ref, op)
        mop = dict(op)
        if op["op"] == "push":
            mop["deltas"] = np.abs(op["deltas"])
        m = apply_ref(mag, mop)
        if op["op"] == "pull":
            assert np.all(np.abs(got - want) <= RTOL * m + 1e-30)
    compare_full_state(pm, ref, K, W, exact=False, mag=mag)
    pm.close()
