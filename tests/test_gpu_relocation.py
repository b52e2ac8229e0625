"""GPU parity of the relocation mode (Sec. 4.1, App. B.2.4) against the CPU oracle.

The CUDA path runs with relocate=1 through the C ABI and the oracle with relocation=True on the same
seeded call sequences.  Bit-exact: owners, replica key sets, refcounts, pulled rows and, with dyadic
deltas (exact sums in any order), every stored value; the counts of created and destroyed replicas
and of relocations.  Gaussian deltas: within 1e-5 of the magnitude bound, as for always-replicate
(the only new rounding is the order of two pending rows merged into one key in the same advance).
The paper's scenarios (Fig. 4b-d, Fig. 10a) run on the GPU as well.
"""
import numpy as np
import pytest
import torch

from oracle import ParameterManagerOracle
from tests.seqgen import dyadic_init, random_sequence
from tests.test_gpu_store import RTOL, apply_gpu, apply_ref, compare_full_state, dev
from tests.test_oracle_relocation import expected_owner, expected_replica, figure_scenarios, ticks

pytestmark = pytest.mark.gpu


def make_pair(gpu_lib, K, D, W, init, capacity=0):
    pm = gpu_lib.ParameterManager(K, D, W, replica_capacity=capacity,
                                  init_values=torch.from_numpy(init).cuda(), relocate=True)
    ref = ParameterManagerOracle(K, D, W, init, relocation=True)
    return pm, ref


def compare_counts(pm, ref):
    st = pm.stats()
    assert (st["created"], st["destroyed"], st["relocations"]) == (ref.created, ref.destroyed, ref.relocations)


CASES = [
    # K, D, W, max_batch, n_ops
    (40, 4, 3, 12, 220),
    (300, 16, 4, 700, 80),
    (5000, 64, 3, 6000, 40),
    (900, 200, 2, 2500, 30),
    (7, 4, 32, 9, 240),          # every worker slot, keys shared by many workers
]


@pytest.mark.parametrize("K,D,W,max_batch,n_ops", CASES)
@pytest.mark.parametrize("seed", [0, 1])
def test_random_sequences_relocation_bit_exact(gpu_lib, K, D, W, max_batch, n_ops, seed):
    init = dyadic_init(K, D, seed + 5)
    pm, ref = make_pair(gpu_lib, K, D, W, init)
    keys = np.arange(K)
    ops = random_sequence(seed * 17 + K + 3, K, D, W, n_ops, max_batch=max_batch)
    for i, op in enumerate(ops):
        got = apply_gpu(pm, op)
        want = apply_ref(ref, op)
        if op["op"] == "pull":
            assert np.array_equal(got, want), f"pull {i}"
        if op["op"] in ("intent", "advance") and K <= 300:
            assert np.array_equal(pm.owners(keys), ref.owners(keys)), f"owners after op {i}"
            for w in range(W):
                assert np.array_equal(pm.replica_keys(w), ref.replica_keys(w)), f"op {i} worker {w}"
    compare_full_state(pm, ref, K, W)
    assert np.array_equal(pm.owners(keys), ref.owners(keys))
    compare_counts(pm, ref)
    pm.sync()
    ref.sync()
    compare_full_state(pm, ref, K, W)
    pm.close()


def test_random_sequence_relocation_gaussian_within_tolerance(gpu_lib):
    K, D, W = 2000, 64, 4
    rng = np.random.default_rng(11)
    init = rng.normal(0, 0.1, size=(K, D)).astype(np.float32)
    pm, ref = make_pair(gpu_lib, K, D, W, init)
    mag = ParameterManagerOracle(K, D, W, np.abs(init), relocation=True)
    for op in random_sequence(2024, K, D, W, 80, max_batch=3000, gaussian=True):
        got = apply_gpu(pm, op)
        want = apply_ref(ref, op)
        mop = dict(op)
        if op["op"] == "push":
            mop["deltas"] = np.abs(op["deltas"])
        m = apply_ref(mag, mop)
        if op["op"] == "pull":
            assert np.all(np.abs(got - want) <= RTOL * m + 1e-30)
    compare_full_state(pm, ref, K, W, exact=False, mag=mag)
    assert np.array_equal(pm.owners(np.arange(K)), ref.owners(np.arange(K)))
    pm.close()


@pytest.mark.parametrize("sc", figure_scenarios(), ids=lambda s: s["name"])
def test_figure_scenarios_on_gpu(gpu_lib, sc):
    W = 4
    pm = gpu_lib.ParameterManager(1, 4, W, replica_capacity=8, relocate=True)
    for node in range(W):
        for n, start, length in sc["intent"]:
            if n == node:
                pm.intent(node, dev([0]), ticks(start), ticks(start) + ticks(length))

    def check(t):
        where = f"{sc['name']} ({sc['cite']}) at t={t / 10}"
        assert pm.owners(np.array([0]))[0] == expected_owner(sc, t), where
        for node in range(W):
            assert (pm.replica_keys(node).tolist() == [0]) == expected_replica(sc, node, t), f"{where} node {node}"

    check(0)
    for t in range(1, ticks(sc["horizon"])):
        for node in range(W):
            pm.advance_clock(node)
        check(t)
    pm.wait()
    pm.close()


def test_always_replicate_reports_no_owner(gpu_lib):
    pm = gpu_lib.ParameterManager(8, 4, 2)
    pm.intent(0, dev([1, 2]), 0, 3)
    assert pm.owners(np.arange(8)).tolist() == [-1] * 8
    assert pm.replica_keys(0).tolist() == [1, 2] and pm.stats()["relocations"] == 0
    pm.close()
