"""Pins of the oracle's versioned refresh (App. B.1.2: holders receive only updates they have not seen).

* exact arithmetic: with dyadic values every sum is exact, so skipping a refresh must change nothing; the
  versioned and the full refresh give identical pulls and stores on random call sequences, in every placement
  and timing mode;
* fp32: a hand-built case where the holder's own rounding and main's differ (the holder keeps its value), and
  the two ways a foreign write forces the refresh (a write without a replica, a destroyed replica);
* gaussian sequences: the versioned refresh stays within fp32 rounding of the full one.
"""
import numpy as np
import pytest

from oracle import ParameterManagerOracle
from tests.seqgen import dyadic_init, random_sequence
from tests.test_oracle_store import apply


@pytest.mark.parametrize("seed", range(8))
@pytest.mark.parametrize("relocation,timing", [(False, "start"), (True, "start"), (False, "adaptive")])
def test_versioned_refresh_changes_nothing_in_exact_arithmetic(seed, relocation, timing):
    K, D, W = 14, 3, 3
    init = dyadic_init(K, D, seed)
    full = ParameterManagerOracle(K, D, W, init, relocation=relocation, action_timing=timing)
    ver = ParameterManagerOracle(K, D, W, init, relocation=relocation, action_timing=timing, delta_refresh=True)
    for op in random_sequence(seed + 700, K, D, W, 260):
        a, b = apply(full, op), apply(ver, op)
        if op["op"] == "pull":
            assert np.array_equal(a, b)
    for w in range(W):
        ka, va, aa = full.replica_values(w)
        kb, vb, ab = ver.replica_values(w)
        assert np.array_equal(ka, kb) and np.array_equal(va, vb) and np.array_equal(aa, ab)
    assert np.array_equal(full.main, ver.main)
    assert ver.refreshed <= full.refreshed


def test_sole_holder_keeps_its_own_rounding():
    eps = np.float32(2.0 ** -24)
    init = np.ones((1, 1), np.float32)
    for delta_refresh, want_val in ((True, 1.0), (False, 1.0 + 2.0 ** -23)):
        pm = ParameterManagerOracle(1, 1, 1, init, delta_refresh=delta_refresh)
        pm.intent(0, [0], 0, 9)
        for _ in range(2):
            pm.push(0, [0], np.array([[eps]], np.float32))
        # 1 + 2^-24 rounds to 1 (ties to even) twice; the pending sum 2^-23 is exact
        assert pm.pull(0, [0]).tolist() == [[1.0]]
        pm.sync()
        assert pm.read_main([0]).tolist() == [[1.0 + 2.0 ** -23]]
        assert pm.pull(0, [0]).tolist() == [[want_val]]
        assert pm.refreshed == (0 if delta_refresh else 1)


@pytest.mark.parametrize("foreign", ["write_without_replica", "destroyed_replica", "second_holder"])
def test_foreign_updates_force_the_refresh(foreign):
    init = np.zeros((2, 2), np.float32)
    pm = ParameterManagerOracle(2, 2, 2, init, delta_refresh=True)
    pm.intent(0, [0], 0, 9)
    pm.push(0, [0], np.full((1, 2), 0.5, np.float32))
    if foreign == "write_without_replica":
        pm.push(1, [0], np.full((1, 2), 0.25, np.float32))       # worker 1 holds no replica: main
    elif foreign == "destroyed_replica":
        pm.intent(1, [0], 0, 1)
        pm.push(1, [0], np.full((1, 2), 0.25, np.float32))
        pm.advance_clock(1)                                      # its replica is destroyed: main += 0.25
    else:
        pm.intent(1, [0], 0, 9)
        pm.push(1, [0], np.full((1, 2), 0.25, np.float32))
    pm.sync()
    assert pm.read_main([0]).tolist() == [[0.75, 0.75]]
    assert pm.pull(0, [0]).tolist() == [[0.75, 0.75]]            # refreshed: sees the other worker's 0.25
    assert pm.refreshed == (2 if foreign == "second_holder" else 1)
    # the next sync with no foreign write skips the refresh
    pm.push(0, [0], np.full((1, 2), 0.125, np.float32))
    if foreign == "second_holder":
        pm.advance_clock(1)
        pm.advance_clock(1)
        for _ in range(8):
            pm.advance_clock(1)                                  # worker 1's window ends: a destroy
    before = pm.refreshed
    pm.sync()
    assert pm.pull(0, [0]).tolist() == [[0.875, 0.875]]
    assert pm.refreshed == before + (1 if foreign == "second_holder" else 0)


def test_gaussian_sequences_stay_within_rounding_of_the_full_refresh():
    K, D, W = 16, 8, 3
    rng = np.random.default_rng(3)
    init = rng.normal(0, 0.1, size=(K, D)).astype(np.float32)
    full = ParameterManagerOracle(K, D, W, init)
    ver = ParameterManagerOracle(K, D, W, init, delta_refresh=True)
    for op in random_sequence(99, K, D, W, 300, gaussian=True):
        a, b = apply(full, op), apply(ver, op)
        if op["op"] == "pull":
            assert np.allclose(a, b, rtol=1e-5, atol=1e-6)
    assert np.allclose(full.main, ver.main, rtol=1e-5, atol=1e-6)
