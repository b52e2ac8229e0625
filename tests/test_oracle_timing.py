"""Pins of the oracle's action timing (Sec. 4.2, Algorithm 1; Sec. 5.8's immediate-action ablation).

* the Poisson quantile against scipy's (a different implementation of the same definition), and its
  closed-form corners;
* the rate estimate against the closed form of the smoothing recursion, the no-update rule for rounds in
  which the worker did not advance, and the max(estimate, Delta) heuristic;
* action timing in the parameter manager: which intents a round acts on (the bound from the pinned
  quantile), that acting early only moves an intent's start, brute-force active sets for acting on
  signal, and the dyadic sum invariant in every timing mode.
"""
import math

import numpy as np
import pytest

from oracle import ParameterManagerOracle
from oracle.timing import LAMBDA0, P, RateEstimate, poisson_quantile
from tests.seqgen import dyadic_init, random_sequence
from tests.test_oracle_store import apply

scipy_stats = pytest.importorskip("scipy.stats")


@pytest.mark.parametrize("lam", [0.05, 0.5, 1.0, 2.0, 2.8, 7.3, 20.0, 64.0, 333.3, 2000.0])
@pytest.mark.parametrize("p", [0.01, 0.5, 0.9, 0.99, 0.9999])
def test_poisson_quantile_matches_scipy(lam, p):
    assert poisson_quantile(lam, p) == int(scipy_stats.poisson.ppf(p, lam))


def test_poisson_quantile_corners():
    # P(X = 0) = exp(-lam): any p up to it gives 0, just above it 1
    for lam in (0.1, 1.0, 5.0):
        assert poisson_quantile(lam, math.exp(-lam) * (1 - 1e-12)) == 0
        assert poisson_quantile(lam, math.exp(-lam) * (1 + 1e-9)) == 1
    # non-decreasing in lam and in p
    qs = [poisson_quantile(lam, P) for lam in np.linspace(0.5, 50, 60)]
    assert all(a <= b for a, b in zip(qs, qs[1:]))
    qs = [poisson_quantile(10.0, p) for p in (0.1, 0.5, 0.9, 0.99, 0.9999)]
    assert all(a <= b for a, b in zip(qs, qs[1:]))
    with pytest.raises(ValueError):
        poisson_quantile(0.0, 0.5)


def test_rate_estimate_closed_form():
    # a worker advancing d clocks per round: est_t = d + (est_0 - d)(1 - alpha)^t
    for d in (1, 3):
        r = RateEstimate()
        for t in range(1, 40):
            b = r.round(d * t)
            want = d + (LAMBDA0 - d) * 0.9 ** t
            assert abs(r.est - want) <= 1e-12 * want
            assert b == int(scipy_stats.poisson.ppf(P, 2 * max(want, d)))


def test_rate_estimate_keeps_its_value_while_paused_and_follows_bursts():
    r = RateEstimate()
    r.round(1)
    est = r.est
    assert est == pytest.approx(0.9 * LAMBDA0 + 0.1)
    for _ in range(5):                       # no clocks: no update (Sec. 4.2)
        assert r.round(1) == int(scipy_stats.poisson.ppf(P, 2 * est))
        assert r.est == est
    # a burst of 50 clocks: the bound follows the burst at once, not the smoothed estimate
    b = r.round(51)
    assert r.est == pytest.approx(0.9 * est + 5.0)
    assert b == int(scipy_stats.poisson.ppf(P, 100.0))


def test_adaptive_round_acts_on_intents_inside_the_bound():
    pm = ParameterManagerOracle(4, 2, 1, np.zeros((4, 2), np.float32), action_timing="adaptive")
    b0 = int(scipy_stats.poisson.ppf(P, 2 * LAMBDA0))      # first round at clock 0: Delta = 0, est = 10
    pm.intent(0, [0], 5, 6)
    pm.intent(0, [1], b0 - 1, b0)
    pm.intent(0, [2], b0, b0 + 1)                           # starts exactly at the bound: not yet
    assert pm.replica_keys(0).tolist() == []                # nothing acts before a round
    pm.sync()
    assert pm.replica_keys(0).tolist() == [0, 1]
    assert pm.refcounts(0, [0, 1, 2]).tolist() == [1, 1, 0]
    for _ in range(6):
        pm.advance_clock(0)
    assert pm.replica_keys(0).tolist() == [1]              # key 0's window [5, 6) ended on time
    while pm.clock[0] < b0:
        pm.advance_clock(0)
    assert pm.replica_keys(0).tolist() == [2]              # no later round: key 2 starts at its start


def test_signal_mode_acts_when_signalled():
    pm = ParameterManagerOracle(4, 2, 2, np.arange(8, dtype=np.float32).reshape(4, 2), action_timing="signal")
    pm.intent(0, [3], 4, 6)
    assert pm.replica_keys(0).tolist() == [3]
    pm.push(0, [3], np.ones((1, 2), np.float32))
    assert pm.read_main([3]).tolist() == [[6.0, 7.0]]       # the write went to the early replica
    for _ in range(6):
        pm.advance_clock(0)
    assert pm.replica_keys(0).tolist() == []
    assert pm.read_main([3]).tolist() == [[7.0, 8.0]]       # merged when the window closed at 6


@pytest.mark.parametrize("seed", range(10))
def test_signal_mode_active_sets_by_brute_force(seed):
    K, D, W = 12, 2, 3
    pm = ParameterManagerOracle(K, D, W, dyadic_init(K, D, seed), action_timing="signal")
    log = []
    for op in random_sequence(seed + 900, K, D, W, 200, max_batch=8):
        if op["op"] == "intent":
            c = pm.clock[op["w"]]
            if op["end"] > op["start"]:          # an empty window stays a no-op
                log.append((op["w"], set(int(k) for k in op["keys"]), min(op["start"], c), op["end"]))
        apply(pm, op)
        for w in range(W):
            c = pm.clock[w]
            want = set()
            for ww, keys, s, e in log:
                if ww == w and s <= c < e:
                    want |= keys
            assert set(pm.replica_keys(w).tolist()) == want


@pytest.mark.parametrize("timing", ["start", "adaptive", "signal"])
@pytest.mark.parametrize("relocation", [False, True])
def test_sum_invariant_in_every_timing_mode(timing, relocation):
    K, D, W = 16, 4, 3
    init = dyadic_init(K, D, 7)
    pm = ParameterManagerOracle(K, D, W, init, relocation=relocation, action_timing=timing)
    total = init.astype(np.float64).copy()
    for op in random_sequence(4242, K, D, W, 300, max_ahead=12):
        if op["op"] == "push":
            np.add.at(total, np.asarray(op["keys"], dtype=np.int64), op["deltas"].astype(np.float64))
        apply(pm, op)
    pm.sync()
    assert np.array_equal(pm.main.astype(np.float64), total)
    for w in range(W):
        ks, val, acc = pm.replica_values(w)
        assert np.array_equal(val, pm.main[ks]) and not acc.any()
