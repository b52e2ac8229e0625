"""Push plans (adapm_intent): a push with the keys of its worker's active intent groups its rows by
the sort made for that intent instead of sorting again; a push with other keys sorts.  Either way the
result is the oracle's: bit-exact with dyadic values, whose sums are exact in any order.  The
library's counters say which path ran (planned_pushes: a plan was checked; plan_misses: its keys
differed)."""
import dataclasses

import numpy as np
import pytest
import torch

from oracle import ParameterManagerOracle, steps
from synth import workloads as wl
from synth.hashgen import init_rows_np
from tests.seqgen import dyadic_init

pytestmark = pytest.mark.gpu


def dyadic_rows(rng, n, D):
    return (rng.integers(-64, 65, size=(n, D)) * 2.0 ** -10).astype(np.float32)


def hot_keys(rng, K, n):
    k = rng.integers(0, K, size=n)
    k[rng.random(n) < 0.25] = 7                   # one key over many push chunks
    return k


def check_same(pm, ref, K, W):
    allk = np.arange(K)
    assert np.array_equal(pm.read_main(allk), ref.read_main(allk))
    for w in range(W):
        ks, val, acc = ref.replica_values(w)
        assert np.array_equal(pm.replica_keys(w), ks)
        gv, ga, has = pm.replica_rows(w, ks)
        assert has.all() and np.array_equal(gv, val) and np.array_equal(ga, acc)


@pytest.mark.parametrize("K,D,n", [(5000, 32, 3000), (200000, 64, 70000)])
def test_push_with_the_intents_keys_uses_its_plan(gpu_lib, K, D, n):
    W = 2
    rng = np.random.default_rng(n)
    init = dyadic_init(K, D, 3)
    pm = gpu_lib.ParameterManager(K, D, W, init_values=torch.from_numpy(init).cuda())
    ref = ParameterManagerOracle(K, D, W, init)
    for c in range(3):
        keys = [hot_keys(rng, K, n) for _ in range(W)]
        for w in range(W):
            kd = torch.as_tensor(keys[w], device="cuda")
            pm.intent(w, kd, c + 1, c + 2)
            ref.intent(w, keys[w], c + 1, c + 2)
            pm.advance_clock(w)
            ref.advance_clock(w)
            d = dyadic_rows(rng, n, D)
            pm.push(w, kd, torch.from_numpy(d).cuda())
            ref.push(w, keys[w], d)
        pm.sync()
        ref.sync()
        pm.wait()
        check_same(pm, ref, K, W)
    st = pm.stats()
    assert st["planned_pushes"] == 3 * W and st["plan_misses"] == 0
    pm.close()


def test_push_with_other_keys_sorts_them(gpu_lib):
    K, D, W, n = 3000, 16, 1, 2500
    rng = np.random.default_rng(5)
    init = dyadic_init(K, D, 4)
    pm = gpu_lib.ParameterManager(K, D, W, init_values=torch.from_numpy(init).cuda())
    ref = ParameterManagerOracle(K, D, W, init)
    a, b = hot_keys(rng, K, n), rng.integers(0, K, size=n)
    b[:10] = a[:10]
    for api, k in ((pm, torch.as_tensor(a, device="cuda")), (ref, a)):
        api.intent(0, k, 1, 3)
        api.advance_clock(0)
    for keys in (b, a, b[::-1].copy()):          # other keys, the intent's, a permutation of other keys
        d = dyadic_rows(rng, n, D)
        pm.push(0, torch.as_tensor(keys, device="cuda"), torch.from_numpy(d).cuda())
        ref.push(0, keys, d)
        pm.wait()
        check_same(pm, ref, K, W)
    st = pm.stats()
    assert st["planned_pushes"] == 3 and st["plan_misses"] == 2
    pm.close()


def test_newest_active_intent_is_the_plan(gpu_lib):
    """Overlapping windows (span 4, a new intent every clock): the push of clock c uses the intent
    signalled for clock c, the newest whose window holds c."""
    K, D, n, span = 20000, 16, 4000, 4
    rng = np.random.default_rng(9)
    init = dyadic_init(K, D, 5)
    pm = gpu_lib.ParameterManager(K, D, 1, init_values=torch.from_numpy(init).cuda())
    ref = ParameterManagerOracle(K, D, 1, init)
    keys = {c: hot_keys(rng, K, n) for c in range(8)}
    for api, cv in ((pm, lambda x: torch.as_tensor(x, device="cuda")), (ref, lambda x: x)):
        api.intent(0, cv(keys[0]), 0, span)
    for c in range(6):
        for api, cv in ((pm, lambda x: torch.as_tensor(x, device="cuda")), (ref, lambda x: x)):
            api.intent(0, cv(keys[c + 1]), c + 1, c + 1 + span)
        d = dyadic_rows(rng, n, D)
        pm.push(0, torch.as_tensor(keys[c], device="cuda"), torch.from_numpy(d).cuda())
        ref.push(0, keys[c], d)
        for api in (pm, ref):
            api.advance_clock(0)
        pm.sync()
        ref.sync()
    pm.wait()
    check_same(pm, ref, K, 1)
    st = pm.stats()
    assert st["planned_pushes"] == 6 and st["plan_misses"] == 0
    pm.close()


def test_intent_keys_from_host_memory(gpu_lib):
    K, D, n = 8000, 16, 5000
    rng = np.random.default_rng(11)
    init = dyadic_init(K, D, 6)
    pm = gpu_lib.ParameterManager(K, D, 2, init_values=torch.from_numpy(init).cuda())
    ref = ParameterManagerOracle(K, D, 2, init)
    pinned = torch.from_numpy(hot_keys(rng, K, n).astype(np.int32)).pin_memory()
    pageable = hot_keys(rng, K, n)
    pm.intent(0, pinned, 1, 2)
    pm.intent(1, pageable, 1, 2)
    ref.intent(0, pinned.numpy(), 1, 2)
    ref.intent(1, pageable, 1, 2)
    for w, keys in ((0, pinned.numpy()), (1, pageable)):
        pm.advance_clock(w)
        ref.advance_clock(w)
        d = dyadic_rows(rng, n, D)
        pm.push(w, torch.as_tensor(keys.astype(np.int64), device="cuda"), torch.from_numpy(d).cuda())
        ref.push(w, keys, d)
    pm.wait()
    check_same(pm, ref, K, 2)
    st = pm.stats()
    assert st["planned_pushes"] == 2 and st["plan_misses"] == 0
    pm.close()


def test_out_of_range_keys_reported_by_a_planned_push(gpu_lib):
    A = gpu_lib
    K, D, n = 1000, 8, 600
    rng = np.random.default_rng(13)
    pm = A.ParameterManager(K, D, 1)
    keys = rng.integers(0, K, size=n)
    keys[[3, 300]] = K + 5
    kd = torch.as_tensor(keys, device="cuda")
    pm.intent(0, kd, 1, 2)
    with pytest.raises(A.AdaPMError) as e:
        pm.wait()
    assert e.value.status == A.ERANGE
    pm.advance_clock(0)
    pm.push(0, kd, torch.ones((n, D), device="cuda"))
    with pytest.raises(A.AdaPMError) as e:
        pm.wait()
    assert e.value.status == A.ERANGE
    good = np.delete(keys, [3, 300])
    want = np.zeros((K, D), np.float32)
    np.add.at(want, good, 1.0)
    # the replicas hold the pushes until the window closes
    pm.advance_clock(0)
    pm.wait()
    assert np.array_equal(pm.read_main(np.arange(K)), want)
    st = pm.stats()
    assert st["planned_pushes"] == 1 and st["plan_misses"] == 0
    pm.close()


def test_plans_on_and_off_give_the_same_bits(gpu_lib):
    """An MF AdaGrad loop (fused steps push cat(rows, cols), the keys the loop signals) with and
    without plans: identical stores, and every step's push used its plan."""
    cfg = dataclasses.replace(wl.MF, name="mf_small", rows=20000, cols=3000, rank=8, workers=3, batch=4000,
                              lookahead=2, zipf_s=1.1, total_cells=10 ** 7)
    init = init_rows_np(np.arange(cfg.num_keys), cfg.value_len, cfg.rank, cfg.seed, cfg.init_std)
    nclk = 5
    batches = {(w, c): [x.cuda() for x in wl.mf_batch(cfg, w, c)] for w in range(cfg.workers)
               for c in range(nclk + cfg.lookahead + 1)}
    out = []
    for plans in (True, False):
        pm = gpu_lib.ParameterManager(cfg.num_keys, cfg.value_len, cfg.workers,
                                      init_values=torch.from_numpy(init).cuda(), push_plans=plans)
        keys = lambda w, c: torch.cat(batches[(w, c)][:2])  # noqa: E731
        for w in range(cfg.workers):
            for j in range(cfg.lookahead):
                pm.intent(w, keys(w, j), j, j + 1)
        for c in range(nclk):
            for w in range(cfg.workers):
                j = c + cfg.lookahead
                pm.intent(w, keys(w, j), j, j + 1)
                r, co, v = batches[(w, c)]
                pm.mf_step(w, r, co, v, cfg.rank, True, cfg.lr, cfg.eps)
                pm.advance_clock(w)
            pm.sync()
        pm.wait()
        out.append(pm.read_main(np.arange(cfg.num_keys)))
        st = pm.stats()
        assert st["planned_pushes"] == (nclk * cfg.workers if plans else 0) and st["plan_misses"] == 0
        pm.close()
    assert np.array_equal(out[0], out[1])


def test_complex_step_uses_its_plan(gpu_lib):
    cfg = dataclasses.replace(wl.COMPLEX, name="complex_small", entities=3000, relations=6, half_dim=8,
                              workers=1, batch=64, negatives=10, lookahead=1, total_triples=10 ** 5)
    init = init_rows_np(np.arange(cfg.num_keys), cfg.value_len, cfg.theta_dim, cfg.seed, 0.3)
    pm = gpu_lib.ParameterManager(cfg.num_keys, cfg.value_len, 1, init_values=torch.from_numpy(init).cuda())
    ref = ParameterManagerOracle(cfg.num_keys, cfg.value_len, 1, init)
    h, r, t, ng = wl.complex_batch(cfg, 0, 1)
    keys = np.concatenate([h.numpy(), r.numpy(), t.numpy(), ng.numpy().reshape(-1)])
    for api, k in ((pm, torch.as_tensor(keys, device="cuda")), (ref, keys)):
        api.intent(0, k, 1, 2)
        api.advance_clock(0)
    want = steps.complex_step(ref, 0, h.numpy(), r.numpy(), t.numpy(), ng.numpy(), cfg.theta_dim, cfg.lr, cfg.eps)
    loss = torch.zeros(1, dtype=torch.float64, device="cuda")
    pm.complex_step(0, h.cuda(), r.cuda(), t.cuda(), ng.reshape(-1).cuda(), cfg.negatives, cfg.theta_dim, cfg.lr,
                    cfg.eps, loss_out=loss)
    pm.wait()
    assert abs(float(loss.item()) - want) <= 1e-4 * abs(want)
    st = pm.stats()
    assert st["planned_pushes"] == 1 and st["plan_misses"] == 0
    for api in (pm, ref):
        api.advance_clock(0)
    main = pm.read_main(np.arange(cfg.num_keys))
    assert np.max(np.abs(main - ref.main)) <= 1e-5 * np.abs(ref.main).max()
    pm.close()


def test_step_with_other_keys_misses_its_plan(gpu_lib):
    """A training step compares the push keys it writes with its plan's keys: a step on another batch of the
    same size counts one miss, sorts its keys, and gives the bits a run without plans gives."""
    cfg = dataclasses.replace(wl.MF, name="mf_small", rows=5000, cols=800, rank=8, workers=1, batch=1500,
                              lookahead=1, zipf_s=1.1, total_cells=10 ** 6)
    init = init_rows_np(np.arange(cfg.num_keys), cfg.value_len, cfg.rank, cfg.seed, cfg.init_std)
    a = [x.cuda() for x in wl.mf_batch(cfg, 0, 1)]
    b = [x.cuda() for x in wl.mf_batch(cfg, 0, 2)]
    out, losses = [], []
    for plans in (True, False):
        pm = gpu_lib.ParameterManager(cfg.num_keys, cfg.value_len, 1, init_values=torch.from_numpy(init).cuda(),
                                      push_plans=plans)
        pm.intent(0, torch.cat(a[:2]), 1, 3)     # signals batch a ...
        pm.advance_clock(0)
        loss = torch.zeros(1, dtype=torch.float64, device="cuda")
        pm.mf_step(0, b[0], b[1], b[2], cfg.rank, True, cfg.lr, cfg.eps, loss_out=loss)   # ... trains on b
        pm.mf_step(0, a[0], a[1], a[2], cfg.rank, True, cfg.lr, cfg.eps)                  # then on a
        pm.advance_clock(0)
        pm.advance_clock(0)
        pm.wait()
        out.append(pm.read_main(np.arange(cfg.num_keys)))
        losses.append(float(loss.item()))
        st = pm.stats()
        if plans:
            assert st["planned_pushes"] == 2 and st["plan_misses"] == 1
        else:
            assert st["planned_pushes"] == 0
        pm.close()
    assert np.array_equal(out[0], out[1]) and losses[0] == losses[1]


def test_sgns_step_sorts_without_a_plan(gpu_lib):
    """The SGNS step's rows follow its centres, never an intent's key order: it looks up no plan, even when an
    intent of exactly its push's size is active, and sorts."""
    vocab, dim, n, n_ctx, n_neg = 300, 16, 40, 4, 3
    K = 2 * vocab
    rng = np.random.default_rng(5)
    pm = gpu_lib.ParameterManager(K, dim, 1)
    centres = torch.as_tensor(rng.integers(0, vocab, size=n), dtype=torch.int32, device="cuda")
    contexts = torch.as_tensor(rng.integers(0, vocab, size=n * n_ctx), dtype=torch.int32, device="cuda")
    negatives = torch.as_tensor(rng.integers(0, vocab, size=n * n_ctx * n_neg), dtype=torch.int32, device="cuda")
    m = n * (1 + n_ctx * (1 + n_neg))
    pm.intent(0, torch.as_tensor(rng.integers(0, K, size=m), device="cuda"), 0, 2)
    pm.sgns_step(0, centres, contexts, negatives, n_ctx, n_neg, vocab, dim, 0.05)
    pm.wait()
    st = pm.stats()
    assert st["planned_pushes"] == 0 and st["plan_misses"] == 0 and st["push_rows"] == m
    pm.close()


def test_worker_whose_plans_go_unused_stops_getting_them(gpu_lib):
    """After four lists in a row closed with a plan no push took, a worker's intents get no plan, except one
    intent in sixteen (a probe); a probe that a push takes brings plans back.  Results match the oracle."""
    K, D, n = 3000, 8, 400
    rng = np.random.default_rng(21)
    init = dyadic_init(K, D, 8)
    pm = gpu_lib.ParameterManager(K, D, 1, init_values=torch.from_numpy(init).cuda())
    ref = ParameterManagerOracle(K, D, 1, init)
    planned = []
    for c in range(20):   # intents 0..19 (clock c signals clock c + 1); intent 16 is a probe
        keys = hot_keys(rng, K, n)
        for api, cv in ((pm, lambda x: torch.as_tensor(x, device="cuda")), (ref, lambda x: x)):
            api.intent(0, cv(keys), c + 1, c + 2)
            api.advance_clock(0)
        # clocks 1..15 push other keys (the plan goes unused); from clock 17 the signalled ones
        push = keys if c >= 16 else hot_keys(rng, K, n // 2)
        d = dyadic_rows(rng, len(push), D)
        pm.push(0, torch.as_tensor(push, device="cuda"), torch.from_numpy(d).cuda())
        ref.push(0, push, d)
        pm.wait()
        planned.append(pm.stats()["planned_pushes"])
    check_same(pm, ref, K, 1)
    # intents 5..15 were recorded after 4 or more unused plans: none has a plan; intent 16 is a probe and the
    # push of clock 17 takes it
    assert planned[15] == 0 and planned[16] == 1
    # intent 17 was recorded before the probe's list closed (no plan); 18 and 19 have plans again
    assert planned[17] == 1 and planned[18] == 2 and planned[19] == 3
    pm.close()
