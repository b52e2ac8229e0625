"""Pins of the oracle's parameter-manager semantics against things other than itself.

* brute force: active sets and intent counts recomputed by scanning the raw
  log of every Intent call (including the no-op ones) against the window
  definition of Sec. 3;
* invariants: replica sets equal active sets; pulls of keys without a replica
  return main; after a final sync main = init + sum of every pushed row
  (bit-exact with dyadic deltas), and every replica equals main;
* hand-worked scenarios in tests/golden/scenarios.json.
"""
import json
import os

import numpy as np
import pytest

from oracle import OracleError, ParameterManagerOracle
from tests.seqgen import dyadic_init, random_sequence

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "scenarios.json")


def brute_active(log, w, clock):
    """Keys of worker w's Intent calls whose window contains `clock` (Sec. 3)."""
    out = set()
    for (ww, keys, s, e) in log:
        if ww == w and s <= clock < e:
            out |= set(int(k) for k in keys)
    return out


def brute_count(log, w, clock, k):
    return sum(1 for (ww, keys, s, e) in log
               if ww == w and s <= clock < e and k in set(int(x) for x in keys))


def apply(pm, op):
    kind = op["op"]
    if kind == "intent":
        pm.intent(op["w"], op["keys"], op["start"], op["end"])
    elif kind == "advance":
        pm.advance_clock(op["w"])
    elif kind == "pull":
        return pm.pull(op["w"], op["keys"])
    elif kind == "push":
        pm.push(op["w"], op["keys"], op["deltas"])
    elif kind == "sync":
        pm.sync()
    return None


@pytest.mark.parametrize("seed", range(12))
def test_replica_sets_equal_brute_force_active_sets(seed):
    K, D, W = 24, 3, 3
    init = dyadic_init(K, D, seed)
    pm = ParameterManagerOracle(K, D, W, init)
    log = []
    for op in random_sequence(seed, K, D, W, 160):
        if op["op"] == "intent":
            log.append((op["w"], op["keys"], op["start"], op["end"]))
        apply(pm, op)
        for w in range(W):
            want = brute_active(log, w, pm.clock[w])
            assert set(pm.replica_keys(w).tolist()) == want
            ks = np.arange(K)
            got = pm.refcounts(w, ks)
            assert got.tolist() == [brute_count(log, w, pm.clock[w], int(k)) for k in ks]


@pytest.mark.parametrize("seed", range(12))
def test_sum_invariant_dyadic_and_pull_rules(seed):
    K, D, W = 20, 4, 3
    init = dyadic_init(K, D, seed)
    pm = ParameterManagerOracle(K, D, W, init)
    total = init.astype(np.float64).copy()
    for op in random_sequence(seed + 100, K, D, W, 200):
        if op["op"] == "push":
            np.add.at(total, np.asarray(op["keys"], dtype=np.int64), op["deltas"].astype(np.float64))
        out = apply(pm, op)
        if op["op"] == "pull":
            # keys without a replica read the main copy (Sec. 4 / Sec. 5.1)
            reps = set(pm.replica_keys(op["w"]).tolist())
            for i, k in enumerate(np.asarray(op["keys"]).tolist()):
                if k not in reps:
                    assert np.array_equal(out[i], pm.main[k])
        if op["op"] == "sync":
            for w in range(W):
                ks, val, acc = pm.replica_values(w)
                assert np.array_equal(val, pm.main[ks])
                assert not acc.any()
    pm.sync()
    assert np.array_equal(pm.main.astype(np.float64), total)
    for w in range(W):
        ks, val, _ = pm.replica_values(w)
        assert np.array_equal(pm.pull(w, ks), pm.main[ks])


def test_sum_invariant_gaussian_within_fp64_reference():
    K, D, W = 16, 8, 4
    rng = np.random.default_rng(5)
    init = rng.normal(0, 0.1, size=(K, D)).astype(np.float32)
    pm = ParameterManagerOracle(K, D, W, init)
    total = init.astype(np.float64).copy()
    for op in random_sequence(77, K, D, W, 300, gaussian=True):
        if op["op"] == "push":
            np.add.at(total, np.asarray(op["keys"], dtype=np.int64), op["deltas"].astype(np.float64))
        apply(pm, op)
    pm.sync()
    assert np.allclose(pm.main, total, rtol=1e-5, atol=1e-6)


def test_golden_scenarios():
    with open(GOLDEN) as f:
        g = json.load(f)
    for sc in g["scenarios"]:
        pm = ParameterManagerOracle(g["num_keys"], g["value_len"], g["num_workers"],
                                    np.array(g["init"], dtype=np.float32))
        for i, st in enumerate(sc["steps"]):
            where = f"{sc['name']} step {i} ({st['op']})"
            op = st["op"]
            if op == "intent":
                pm.intent(st["w"], st["keys"], st["start"], st["end"])
            elif op == "advance":
                pm.advance_clock(st["w"])
            elif op == "push":
                pm.push(st["w"], st["keys"], np.array(st["deltas"], dtype=np.float32))
            elif op == "sync":
                pm.sync()
            elif op == "pull":
                assert pm.pull(st["w"], st["keys"]).tolist() == st["expect"], where
            elif op == "main":
                assert pm.read_main(st["keys"]).tolist() == st["expect"], where
            elif op == "replica_keys":
                assert pm.replica_keys(st["w"]).tolist() == st["expect"], where
            elif op == "refcounts":
                assert pm.refcounts(st["w"], st["keys"]).tolist() == st["expect"], where
            else:
                raise AssertionError(op)


def test_rejects_bad_arguments():
    pm = ParameterManagerOracle(4, 2, 2, np.zeros((4, 2), np.float32))
    with pytest.raises(OracleError):
        pm.pull(2, [0])
    with pytest.raises(OracleError):
        pm.pull(0, [4])
    with pytest.raises(OracleError):
        pm.intent(0, [0, 9], 0, 1)
    with pytest.raises(OracleError):
        pm.push(1, [-1], np.zeros((1, 2), np.float32))
    # nothing changed
    assert pm.replica_keys(0).tolist() == [] and not pm.main.any()


def test_empty_calls_are_noops():
    pm = ParameterManagerOracle(4, 2, 1, np.ones((4, 2), np.float32))
    pm.intent(0, [], 0, 5)
    pm.push(0, [], np.zeros((0, 2), np.float32))
    assert pm.pull(0, []).shape == (0, 2)
    pm.sync()
    assert (pm.main == 1).all() and pm.replica_keys(0).tolist() == []
