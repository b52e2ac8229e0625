"""GPU parity of action timing (Sec. 4.2, Algorithm 1; the immediate-action variant of Sec. 5.8).

The CUDA path (host controller in the library, events on the GPU) and the oracle run the same seeded call
sequences with action_timing "adaptive" or "signal", with and without relocation.  Intents are signalled up to
40 clocks ahead, so the Poisson bound of each round leaves some for later rounds.  Bit-exact with dyadic deltas:
replica sets, refcounts (which count an intent from the round that acted on it), owners, pulls and every stored
value; the MF loop's losses within 1e-4 with adaptive timing.
"""
import numpy as np
import pytest
import torch

from oracle import ParameterManagerOracle
from tests.seqgen import dyadic_init, random_sequence
from tests.test_gpu_store import apply_gpu, apply_ref, compare_full_state

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("timing", ["adaptive", "signal"])
@pytest.mark.parametrize("relocate", [False, True])
@pytest.mark.parametrize("K,D,W,max_batch,n_ops", [(40, 4, 3, 12, 300), (3000, 64, 4, 4000, 60)])
def test_random_sequences_with_action_timing_bit_exact(gpu_lib, timing, relocate, K, D, W, max_batch, n_ops):
    init = dyadic_init(K, D, 21)
    pm = gpu_lib.ParameterManager(K, D, W, init_values=torch.from_numpy(init).cuda(), relocate=relocate,
                                  action_timing=timing)
    ref = ParameterManagerOracle(K, D, W, init, relocation=relocate, action_timing=timing)
    keys = np.arange(K)
    ops = random_sequence(K + W + n_ops, K, D, W, n_ops, max_batch=max_batch, max_ahead=40, max_span=6)
    for i, op in enumerate(ops):
        got = apply_gpu(pm, op)
        want = apply_ref(ref, op)
        if op["op"] == "pull":
            assert np.array_equal(got, want), f"pull {i}"
        if op["op"] in ("intent", "advance", "sync") and K <= 40:
            for w in range(W):
                assert np.array_equal(pm.replica_keys(w), ref.replica_keys(w)), f"op {i} ({op['op']}) worker {w}"
                assert np.array_equal(pm.refcounts(w, keys), ref.refcounts(w, keys)), f"op {i} worker {w}"
    compare_full_state(pm, ref, K, W)
    assert np.array_equal(pm.owners(keys), ref.owners(keys))
    pm.sync()
    ref.sync()
    compare_full_state(pm, ref, K, W)
    pm.close()


def test_adaptive_timing_custom_parameters(gpu_lib):
    # a small initial rate and quantile: the first round acts only on intents starting within Q(2, 0.5) = 2
    K, D, W = 8, 4, 1
    init = dyadic_init(K, D, 3)
    kw = dict(timing_alpha=0.5, timing_p=0.5, timing_lambda0=1.0)
    pm = gpu_lib.ParameterManager(K, D, W, init_values=torch.from_numpy(init).cuda(), action_timing="adaptive",
                                  **kw)
    ref = ParameterManagerOracle(K, D, W, init, action_timing="adaptive", **kw)
    dev = lambda k: torch.as_tensor(np.asarray(k, dtype=np.int64), device="cuda")  # noqa: E731
    for k, s in enumerate([1, 2, 3, 5]):
        pm.intent(0, dev([k]), s, s + 2)
        ref.intent(0, [k], s, s + 2)
    for step in range(6):
        pm.sync()
        ref.sync()
        assert pm.replica_keys(0).tolist() == ref.replica_keys(0).tolist(), step
        pm.advance_clock(0)
        ref.advance_clock(0)
    pm.wait()
    pm.close()
