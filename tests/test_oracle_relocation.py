"""Pins of the oracle's relocation mode (Sec. 4.1, App. B.2.4) against things other than itself.

* the intent scenarios of Fig. 4b-d and Fig. 10a (tests/golden/relocation_figures.json): the owner and the
  replica intervals that the paper draws, at every clock;
* brute force: after every call of a random sequence, the owner is recomputed from the raw call log by the
  rule as the paper states it (whenever exactly one worker has active intent, that worker holds the
  parameter) and the replica sets must be the active sets minus owned keys;
* closed forms: a sole active worker reads other workers' writes at once (no staleness for non-replicated
  parameters, Sec. 5.1), where always-replicate hides them until a sync; relocation to a replica holder
  merges its pending updates before any sync; a single worker never holds a replica;
* the sum invariant after a final sync, bit-exact with dyadic deltas.
"""
import json
import os

import numpy as np
import pytest

from oracle import ParameterManagerOracle
from tests.seqgen import dyadic_init, random_sequence
from tests.test_oracle_store import apply, brute_active

FIGS = os.path.join(os.path.dirname(__file__), "golden", "relocation_figures.json")
SCALE = 10   # figure units -> clocks


def figure_scenarios():
    with open(FIGS) as f:
        return json.load(f)["scenarios"]


def ticks(x):
    return int(round(x * SCALE))


def expected_owner(sc, t):
    own = None
    for start, node in sc["owner"]:
        if ticks(start) <= t:
            own = node
    return own


def expected_replica(sc, node, t):
    return any(ticks(s) <= t < ticks(e) for s, e in sc["replicas"][str(node)])


def run_figure(sc, relocation=True):
    """Signal every intent at clock 0 (node order), then advance all nodes one clock at a time.

    Yields (t, pm) once every node's clock equals t."""
    W = 4
    pm = ParameterManagerOracle(1, 2, W, np.zeros((1, 2), np.float32), relocation=relocation)
    for node in range(W):
        for n, start, length in sc["intent"]:
            if n == node:
                pm.intent(node, [0], ticks(start), ticks(start) + ticks(length))
    yield 0, pm
    for t in range(1, ticks(sc["horizon"])):
        for node in range(W):
            pm.advance_clock(node)
        yield t, pm


@pytest.mark.parametrize("sc", figure_scenarios(), ids=lambda s: s["name"])
def test_figure_scenarios(sc):
    for t, pm in run_figure(sc):
        where = f"{sc['name']} ({sc['cite']}) at t={t / SCALE}"
        assert pm.owners([0])[0] == expected_owner(sc, t), where
        for node in range(4):
            assert (0 in pm.replica_keys(node).tolist()) == expected_replica(sc, node, t), f"{where} node {node}"


def test_figure_10a_is_not_the_rejected_rule():
    # Fig. 10b would relocate to node 1 once node 0's intent expires at 3
    sc = {s["name"]: s for s in figure_scenarios()}["relocate_only_when_exactly_one_node_has_active_intent"]
    for t, pm in run_figure(sc):
        if ticks(3) <= t < ticks(8):
            assert pm.owners([0])[0] == 0


def test_always_replicate_mode_replicates_every_active_intent():
    # the same scenario without relocation: every active intent has a replica, nothing is owned
    sc = {s["name"]: s for s in figure_scenarios()}["hotspot"]
    for t, pm in run_figure(sc, relocation=False):
        for node in range(4):
            active = any(n == node and ticks(s) <= t < ticks(s) + ticks(ln) for n, s, ln in sc["intent"])
            assert (0 in pm.replica_keys(node).tolist()) == active
        assert pm.owners([0])[0] == -1


@pytest.mark.parametrize("seed", range(16))
def test_owner_and_replicas_equal_brute_force(seed):
    K, D, W = 12, 2, 3
    pm = ParameterManagerOracle(K, D, W, dyadic_init(K, D, seed), relocation=True)
    log = []
    owner = [-1] * K
    for op in random_sequence(seed + 300, K, D, W, 240, max_batch=8):
        if op["op"] == "intent":
            log.append((op["w"], op["keys"], op["start"], op["end"]))
        apply(pm, op)
        active = [brute_active(log, w, pm.clock[w]) for w in range(W)]
        for k in range(K):
            holders = [w for w in range(W) if k in active[w]]
            if len(holders) == 1:
                owner[k] = holders[0]
        assert pm.owners(np.arange(K)).tolist() == owner
        for w in range(W):
            want = sorted(k for k in active[w] if owner[k] != w)
            assert pm.replica_keys(w).tolist() == want


@pytest.mark.parametrize("seed", range(12))
def test_sum_invariant_dyadic_relocation(seed):
    K, D, W = 16, 4, 3
    init = dyadic_init(K, D, seed)
    pm = ParameterManagerOracle(K, D, W, init, relocation=True)
    total = init.astype(np.float64).copy()
    for op in random_sequence(seed + 500, K, D, W, 220):
        if op["op"] == "push":
            np.add.at(total, np.asarray(op["keys"], dtype=np.int64), op["deltas"].astype(np.float64))
        out = apply(pm, op)
        if op["op"] == "pull":
            reps = set(pm.replica_keys(op["w"]).tolist())
            for i, k in enumerate(np.asarray(op["keys"]).tolist()):
                if k not in reps:
                    assert np.array_equal(out[i], pm.main[k])
    pm.sync()
    assert np.array_equal(pm.main.astype(np.float64), total)
    for w in range(W):
        ks, val, acc = pm.replica_values(w)
        assert np.array_equal(val, pm.main[ks]) and not acc.any()


def test_sole_active_worker_sees_other_writes_at_once():
    init = np.array([[1.0, 2.0], [3.0, 4.0]], np.float32)
    for relocation, want_before_sync in ((True, [2.0, 3.0]), (False, [1.0, 2.0])):
        pm = ParameterManagerOracle(2, 2, 2, init, relocation=relocation)
        pm.intent(0, [0], 0, 5)
        assert pm.replica_keys(0).tolist() == ([] if relocation else [0])
        pm.push(1, [0], np.array([[1.0, 1.0]], np.float32))       # worker 1: no intent, writes main
        assert pm.pull(0, [0]).tolist() == [want_before_sync]
        pm.sync()
        assert pm.pull(0, [0]).tolist() == [[2.0, 3.0]]


def test_relocation_to_a_replica_holder_merges_its_updates():
    init = np.array([[1.0, 1.0]], np.float32)
    pm = ParameterManagerOracle(1, 2, 2, init, relocation=True)
    pm.intent(0, [0], 0, 2)          # sole: worker 0 owns key 0
    pm.intent(1, [0], 0, 5)          # second: worker 1 gets a replica
    assert pm.owners([0]).tolist() == [0] and pm.replica_keys(1).tolist() == [0]
    pm.push(1, [0], np.array([[0.5, 0.25]], np.float32))
    pm.push(0, [0], np.array([[2.0, 2.0]], np.float32))        # the owner writes main directly
    assert pm.pull(1, [0]).tolist() == [[1.5, 1.25]]            # replica: stale main + own updates
    pm.advance_clock(0)
    pm.advance_clock(0)                                         # worker 0's intent expires
    assert pm.owners([0]).tolist() == [1] and pm.replica_keys(1).tolist() == []
    assert pm.read_main([0]).tolist() == [[3.5, 3.25]]          # 1 + 2 + 0.5, before any sync
    assert pm.pull(1, [0]).tolist() == [[3.5, 3.25]]
    assert (pm.created, pm.destroyed, pm.relocations) == (1, 1, 2)


def test_single_worker_never_holds_a_replica():
    K, D = 10, 2
    pm = ParameterManagerOracle(K, D, 1, dyadic_init(K, D, 3), relocation=True)
    for op in random_sequence(41, K, D, 1, 150):
        apply(pm, op)
        assert pm.replica_keys(0).tolist() == []
    assert pm.created == 0
