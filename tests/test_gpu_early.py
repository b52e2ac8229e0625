"""GPU parity of early advance events (adapm_advance_clock, Sec. 3 and 4.1).

The refcount events of a worker's next advance are computed at its first
pull, push or training step after an advance, beside the library stream;
the advance then only evicts and creates.  These tests check that this
gives the state the oracle gives, bit for bit with dyadic data, and the
state of the same calls with early events switched off:
  * a loop shaped like the microbenchmark (intent ahead, pull, push,
    advance, sync per clock), where every advance uses its early events;
  * intents recorded or applied between the pull and the advance (the
    early events are undone and the advance runs in full);
  * refcount queries between push and advance (they report the worker's
    current clock);
  * replica capacity running out in an advance that uses early events;
  * the random call sequences of the store tests, early on against off;
  * relocation and adaptive timing, which never use early events.
"""
import numpy as np
import pytest
import torch

from oracle import ParameterManagerOracle
from tests.seqgen import dyadic_init, random_sequence
from tests.test_gpu_store import apply_gpu, apply_ref, compare_full_state, dev

pytestmark = pytest.mark.gpu


def zipf_keys(rng, K, n, s=1.1):
    p = 1.0 / np.arange(1, K + 1) ** s
    return rng.choice(K, size=n, p=p / p.sum())


def loop_ops(seed, K, D, W, clocks, batch, lookahead, span, extra=None):
    """Per clock and worker: intent for clock c + lookahead, pull and push of clock c's keys, advance;
    one sync per clock.  `extra(c, w)` may return ops to insert between the push and the advance."""
    rng = np.random.default_rng(seed)
    keys = {(w, c): zipf_keys(rng, K, batch) for w in range(W) for c in range(clocks + lookahead + 1)}
    ops = []
    for w in range(W):
        for c in range(lookahead):
            ops.append({"op": "intent", "w": w, "keys": keys[(w, c)], "start": c, "end": c + span})
    for c in range(clocks):
        for w in range(W):
            j = c + lookahead
            ops.append({"op": "intent", "w": w, "keys": keys[(w, j)], "start": j, "end": j + span})
            ops.append({"op": "pull", "w": w, "keys": keys[(w, c)]})
            d = (rng.integers(-64, 65, size=(batch, D)) * 2.0 ** -10).astype(np.float32)
            ops.append({"op": "push", "w": w, "keys": keys[(w, c)], "deltas": d})
            if extra is not None:
                ops.extend(extra(c, w, rng))
            ops.append({"op": "advance", "w": w})
        ops.append({"op": "sync"})
    return ops


def run_pair(gpu_lib, K, D, W, ops, init, early=True, oracle=True, **kw):
    pm = gpu_lib.ParameterManager(K, D, W, init_values=torch.from_numpy(init).cuda(), early_events=early, **kw)
    ref = ParameterManagerOracle(K, D, W, init) if oracle else None
    for i, op in enumerate(ops):
        got = apply_gpu(pm, op)
        if ref is not None:
            want = apply_ref(ref, op)
            if op["op"] == "pull":
                assert np.array_equal(got, want), f"pull {i}"
    return pm, ref


def full_state(pm, K, W):
    keys = np.arange(K)
    pm.wait()
    out = {"main": pm.read_main(keys)}
    for w in range(W):
        val, acc, has = pm.replica_rows(w, keys)
        out[w] = (pm.replica_keys(w), pm.refcounts(w, keys), val[has.astype(bool)], acc[has.astype(bool)])
    return out


def assert_same_state(a, b, W):
    assert np.array_equal(a["main"], b["main"])
    for w in range(W):
        for x, y in zip(a[w], b[w]):
            assert np.array_equal(x, y), f"worker {w}"


@pytest.mark.parametrize("K,D,W,batch,lookahead,span", [
    (3000, 64, 3, 700, 1, 1),      # the microbenchmark's shape: windows open at the next clock
    (2000, 200, 2, 500, 2, 2),     # overlapping windows, lists from push plans
    (800, 16, 4, 300, 1, 3),
])
def test_loop_uses_early_events_bit_exact(gpu_lib, K, D, W, batch, lookahead, span):
    clocks = 6
    init = dyadic_init(K, D, 5)
    ops = loop_ops(11 + K, K, D, W, clocks, batch, lookahead, span)
    pm, ref = run_pair(gpu_lib, K, D, W, ops, init)
    st = pm.stats()
    assert st["early_advances"] == clocks * W and st["early_undone"] == 0
    compare_full_state(pm, ref, K, W)
    early = full_state(pm, K, W)
    pm.close()
    pm_off, _ = run_pair(gpu_lib, K, D, W, ops, init, early=False, oracle=False)
    assert pm_off.stats()["early_advances"] == 0
    assert_same_state(early, full_state(pm_off, K, W), W)
    pm_off.close()


def test_intents_between_pull_and_advance_undo_early_events(gpu_lib):
    K, D, W = 1500, 32, 3

    def extra(c, w, rng):
        k = rng.integers(0, K, size=int(rng.integers(1, 200)))
        r = (c + w) % 3
        if r == 0:     # opens at the next clock: the advance's lists differ from the early ones
            return [{"op": "intent", "w": w, "keys": k, "start": c + 1, "end": c + 2}]
        if r == 1:     # active at once: applied now, before the advance
            return [{"op": "intent", "w": w, "keys": k, "start": c, "end": c + 2}]
        return []

    init = dyadic_init(K, D, 7)
    ops = loop_ops(3, K, D, W, 6, 400, 1, 1, extra=extra)
    pm, ref = run_pair(gpu_lib, K, D, W, ops, init)
    st = pm.stats()
    assert st["early_undone"] > 0 and st["early_advances"] > 0
    compare_full_state(pm, ref, K, W)
    pm.close()


def test_refcounts_between_push_and_advance_report_the_current_clock(gpu_lib):
    K, D, W = 600, 8, 2
    init = dyadic_init(K, D, 9)
    ops = loop_ops(21, K, D, W, 5, 250, 1, 1)
    pm = gpu_lib.ParameterManager(K, D, W, init_values=torch.from_numpy(init).cuda())
    ref = ParameterManagerOracle(K, D, W, init)
    keys = np.arange(K)
    for op in ops:
        apply_gpu(pm, op)
        apply_ref(ref, op)
        if op["op"] == "push":
            w = op["w"]
            assert np.array_equal(pm.refcounts(w, keys), ref.refcounts(w, keys))
    assert pm.stats()["early_undone"] > 0
    compare_full_state(pm, ref, K, W)
    pm.close()


def test_capacity_exhausted_in_an_early_advance(gpu_lib):
    """Creations that need more slots than are free fail together (ENOMEM at wait), early or not."""
    K, D, W = 400, 8, 2
    init = dyadic_init(K, D, 13)
    ops = loop_ops(5, K, D, W, 5, 120, 1, 2)

    def run(early):
        pm = gpu_lib.ParameterManager(K, D, W, replica_capacity=90, init_values=torch.from_numpy(init).cuda(),
                                      early_events=early)
        statuses = []
        for op in ops:
            apply_gpu(pm, op)
            if op["op"] == "advance":
                try:
                    pm.wait()
                    statuses.append(0)
                except gpu_lib.AdaPMError as e:
                    statuses.append(e.status)
        return pm, statuses

    pm_on, s_on = run(True)
    pm_off, s_off = run(False)
    assert s_on == s_off and gpu_lib.ENOMEM in s_on
    assert pm_on.stats()["early_advances"] > 0
    assert_same_state(full_state(pm_on, K, W), full_state(pm_off, K, W), W)
    st_on, st_off = pm_on.stats(), pm_off.stats()
    for f in ("live_replicas", "high_water", "created", "destroyed"):
        assert st_on[f] == st_off[f], f
    pm_on.close()
    pm_off.close()


@pytest.mark.parametrize("K,D,W,max_batch,n_ops,seed", [
    (40, 4, 3, 12, 200, 0),
    (300, 16, 4, 700, 80, 1),
    (5000, 64, 3, 6000, 50, 2),
])
def test_random_sequences_early_on_and_off_agree(gpu_lib, K, D, W, max_batch, n_ops, seed):
    init = dyadic_init(K, D, seed)
    ops = random_sequence(seed * 17 + K, K, D, W, n_ops, max_batch=max_batch)
    pm, ref = run_pair(gpu_lib, K, D, W, ops, init)
    compare_full_state(pm, ref, K, W)
    on = full_state(pm, K, W)
    pm.close()
    pm_off, _ = run_pair(gpu_lib, K, D, W, ops, init, early=False, oracle=False)
    assert_same_state(on, full_state(pm_off, K, W), W)
    pm_off.close()


@pytest.mark.parametrize("kw", [{"relocate": True}, {"action_timing": "adaptive"}])
def test_relocation_and_adaptive_timing_never_run_early(gpu_lib, kw):
    K, D, W = 500, 8, 2
    init = dyadic_init(K, D, 3)
    ops = loop_ops(8, K, D, W, 4, 150, 1, 1)
    pm, _ = run_pair(gpu_lib, K, D, W, ops, init, oracle=False, **kw)
    pm.wait()
    st = pm.stats()
    assert st["early_advances"] == 0 and st["early_undone"] == 0
    pm.close()


@pytest.mark.parametrize("host", ["pinned", "pageable"])
def test_host_intent_keys_with_early_events(gpu_lib, host):
    """Intents with host keys (staged copies) in the microbenchmark loop, early events on."""
    K, D, W = 2500, 16, 2
    init = dyadic_init(K, D, 17)
    ops = loop_ops(29, K, D, W, 5, 600, 1, 2)
    pm = gpu_lib.ParameterManager(K, D, W, init_values=torch.from_numpy(init).cuda())
    ref = ParameterManagerOracle(K, D, W, init)
    keep = []   # pinned inputs stay unchanged until adapm_wait; the staged device copies are the library's
    for op in ops:
        if op["op"] == "intent":
            k = torch.from_numpy(np.asarray(op["keys"], dtype=np.int32))
            if host == "pinned":
                k = k.pin_memory()
                keep.append(k)
            pm.intent(op["w"], k, op["start"], op["end"])
        else:
            apply_gpu(pm, op)
        apply_ref(ref, op)
    assert pm.stats()["early_advances"] > 0
    compare_full_state(pm, ref, K, W)
    pm.close()


def test_allocation_free_push_between_early_events_and_the_advance(gpu_lib):
    """The allocation-free push makes no early events of its own (it allocates nothing); the pull before it
    does, and the advance uses them: the same state as the oracle."""
    K, D, W = 2000, 32, 3
    init = dyadic_init(K, D, 23)
    ops = loop_ops(31, K, D, W, 5, 500, 1, 1)
    pm = gpu_lib.ParameterManager(K, D, W, init_values=torch.from_numpy(init).cuda())
    ref = ParameterManagerOracle(K, D, W, init)
    for op in ops:
        if op["op"] == "push":
            pm.push_noalloc(op["w"], dev(op["keys"]), torch.from_numpy(np.ascontiguousarray(op["deltas"])).cuda())
        else:
            got = apply_gpu(pm, op)
            if op["op"] == "pull":
                assert np.array_equal(got, ref.pull(op["w"], op["keys"]))
                continue
        apply_ref(ref, op)
    st = pm.stats()
    assert st["early_advances"] == 5 * W and st["early_undone"] == 0
    compare_full_state(pm, ref, K, W)
    pm.close()
