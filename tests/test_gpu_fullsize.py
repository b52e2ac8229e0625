"""Parity at the full sizes of the workloads, in the bench's launch configuration.

* microbench (100M keys x 64, W=8, 2^20 Zipf(1.1) keys per worker per clock,
  intent span 2), always replicating and with relocation (owners compared
  too): the manager's semantics are separable by key, so the oracle
  replays the whole call sequence restricted to a sample of keys (the hottest
  keys of the batches, random batch keys and keys never touched) and every
  value the GPU holds for those keys is compared bit-exactly (dyadic initial
  values and deltas make every fp32 sum exact in any order).
* MF 10M x 1M rank 100 + AdaGrad: one clock of all 8 workers; the oracle runs
  the same clock on the store restricted to the keys that clock touches.
  Losses within 1e-4, the stored rows within 1e-4 of each block's scale.
* ComplEx 5M and SGNS 700K: worker 0's loss at the first clock depends only on
  the initial store, which the oracle regenerates for the keys of the batch
  (computed in slices); within 1e-4.
"""
import dataclasses

import numpy as np
import pytest
import torch

from oracle import ParameterManagerOracle, driver, steps
from synth import hashgen
from synth import workloads as wl

pytestmark = pytest.mark.gpu


def dev(x):
    return torch.as_tensor(np.asarray(x), device="cuda")


@pytest.mark.parametrize("relocate", [False, True])
def test_micro_full_size_sampled_keys_bit_exact(gpu_lib, relocate):
    cfg = dataclasses.replace(wl.MICRO, span=2)
    K, D, W, B = cfg.num_keys, cfg.value_len, cfg.workers, cfg.batch
    nclk = 3
    keys = {(w, c): wl.micro_keys(cfg, w, c).numpy() for w in range(W) for c in range(nclk + cfg.lookahead + 1)}
    deltas = {(w, c): wl.micro_deltas(cfg, w, c, B, dyadic=True).numpy() for w in range(W) for c in range(nclk)}
    # the store: dyadic values from the counter hash, generated on the GPU
    init = hashgen.init_store_torch(K, D, D, cfg.seed, 0.0, "cuda", kind="dyadic", chunk_rows=1 << 22)
    pm = gpu_lib.ParameterManager(K, D, W, replica_capacity=W * (cfg.span + 1) * B, init_values=init,
                                  relocate=relocate)
    del init
    torch.cuda.empty_cache()
    pulled = {}

    def keys_gpu(w, c):
        return dev(keys[(w, c)].astype(np.int32))

    # the key sample (chosen before the run so that only its pulled rows are kept)
    allk = np.concatenate([keys[(w, c)] for w in range(W) for c in range(nclk + 1)])
    uniq, cnt = np.unique(allk, return_counts=True)
    rng = np.random.default_rng(7)
    hot = uniq[np.argsort(-cnt)[:64]]
    rand = rng.choice(uniq, size=2000, replace=False)
    cold = rng.integers(0, K, size=500)
    sample = np.unique(np.concatenate([hot, rand, cold]))
    masks = {wc: np.isin(k, sample) for wc, k in keys.items()}

    for w in range(W):
        pm.intent(w, keys_gpu(w, 0), 0, cfg.span)
    for c in range(nclk):
        for w in range(W):
            pm.intent(w, keys_gpu(w, c + 1), c + 1, c + 1 + cfg.span)
            pulled[(w, c)] = pm.pull(w, keys_gpu(w, c)).cpu().numpy()[masks[(w, c)]]
            pm.push(w, keys_gpu(w, c), torch.from_numpy(deltas[(w, c)]).cuda())
            pm.advance_clock(w)
        pm.sync()
    pm.wait()

    ref = ParameterManagerOracle(sample.size, D, W,
                                 hashgen.init_rows_np(sample, D, D, cfg.seed, 0.0, kind="dyadic"),
                                 relocation=relocate)

    def restrict(w, c):
        m = masks[(w, c)]
        return m, np.searchsorted(sample, keys[(w, c)][m])

    for w in range(W):
        ref.intent(w, restrict(w, 0)[1], 0, cfg.span)
    for c in range(nclk):
        for w in range(W):
            ref.intent(w, restrict(w, c + 1)[1], c + 1, c + 1 + cfg.span)
            m, rk = restrict(w, c)
            assert np.array_equal(pulled[(w, c)], ref.pull(w, rk)), f"pull w{w} c{c}"
            ref.push(w, rk, deltas[(w, c)][m])
            ref.advance_clock(w)
        ref.sync()
    assert np.array_equal(pm.read_main(sample), ref.main)
    for w in range(W):
        val, acc, has = pm.replica_rows(w, sample)
        rk, rval, racc = ref.replica_values(w)
        assert np.array_equal(np.nonzero(has)[0], rk)
        assert np.array_equal(val[rk], rval) and np.array_equal(acc[rk], racc)
        assert np.array_equal(pm.refcounts(w, sample), ref.refcounts(w, np.arange(sample.size)))
    assert np.array_equal(pm.owners(sample), ref.owners(np.arange(sample.size)))
    pm.close()


def test_mf_full_size_first_clock(gpu_lib):
    cfg = wl.MF
    W, L = cfg.workers, cfg.lookahead
    batches = {(w, c): wl.mf_batch(cfg, w, c) for w in range(W) for c in range(L + 1)}
    init = hashgen.init_store_torch(cfg.num_keys, cfg.value_len, cfg.rank, cfg.seed, cfg.init_std, "cuda",
                                    chunk_rows=1 << 21)
    pm = gpu_lib.ParameterManager(cfg.num_keys, cfg.value_len, W, replica_capacity=W * 4 * cfg.batch,
                                  init_values=init)
    del init
    torch.cuda.empty_cache()

    def keys_of(w, c):
        r, co, _ = batches[(w, c)]
        return np.concatenate([r.numpy(), co.numpy()])

    for w in range(W):
        for j in range(L):
            pm.intent(w, dev(keys_of(w, j).astype(np.int32)), j, j + 1)
    loss = torch.zeros(W, dtype=torch.float64, device="cuda")
    for w in range(W):
        pm.intent(w, dev(keys_of(w, L).astype(np.int32)), L, L + 1)
        r, co, v = batches[(w, 0)]
        pm.mf_step(w, dev(r), dev(co), v.cuda(), cfg.rank, True, cfg.lr, cfg.eps, loss_out=loss[w:w + 1])
        pm.advance_clock(w)
    pm.sync()
    pm.wait()

    # the oracle on the keys this clock reads and writes (batch 0 of every worker)
    touched = np.unique(np.concatenate([keys_of(w, 0) for w in range(W)]))
    ref = ParameterManagerOracle(touched.size, cfg.value_len, W,
                                 hashgen.init_rows_np(touched, cfg.value_len, cfg.rank, cfg.seed, cfg.init_std))
    rel = lambda x: np.searchsorted(touched, x)  # noqa: E731

    def keys_rel(w, c):
        k = keys_of(w, c)
        return rel(k[np.isin(k, touched)])

    def work(w, c):
        r, co, v = batches[(w, c)]
        return steps.mf_step(ref, w, rel(r.numpy()), rel(co.numpy()), v.numpy(), cfg.rank, cfg.lr, True, cfg.eps)

    driver.start(ref, W, L, 1, keys_rel)
    want = driver.clock(ref, W, L, 1, 0, keys_rel, work)
    got = loss.cpu().numpy()
    assert np.all(np.abs(got - want) <= 1e-4 * np.abs(want))
    main = pm.read_main(touched)
    for blk in (slice(0, cfg.rank), slice(cfg.rank, 2 * cfg.rank)):
        assert np.max(np.abs(main[:, blk] - ref.main[:, blk])) <= 1e-4 * np.abs(ref.main[:, blk]).max()
    pm.close()


def _first_loss_gpu(gpu_lib, cfg, keys, run_step, value_len, theta_dim):
    init = hashgen.init_store_torch(cfg.num_keys, value_len, theta_dim, cfg.seed, cfg.init_std, "cuda",
                                    chunk_rows=1 << 20)
    pm = gpu_lib.ParameterManager(cfg.num_keys, value_len, cfg.workers, replica_capacity=4 * len(keys),
                                  init_values=init)
    del init
    torch.cuda.empty_cache()
    pm.intent(0, dev(keys.astype(np.int32)), 0, 1)
    loss = torch.zeros(1, dtype=torch.float64, device="cuda")
    run_step(pm, loss)
    pm.wait()
    pm.close()
    return float(loss.item())


def test_complex_full_size_first_clock_loss(gpu_lib):
    cfg = wl.COMPLEX
    h, r, t, n = (x.numpy() for x in wl.complex_batch(cfg, 0, 0))
    keys = np.concatenate([h, r, t, n.reshape(-1)])

    def run(pm, loss):
        pm.complex_step(0, dev(h), dev(r), dev(t), dev(n.reshape(-1)), cfg.negatives, cfg.theta_dim, cfg.lr,
                        cfg.eps, loss_out=loss)

    got = _first_loss_gpu(gpu_lib, cfg, keys, run, cfg.value_len, cfg.theta_dim)
    td = cfg.theta_dim
    want = 0.0
    for s0 in range(0, h.size, 256):
        sl = slice(s0, s0 + 256)
        rows = lambda k: hashgen.init_rows_np(k.reshape(-1), cfg.value_len, td, cfg.seed, cfg.init_std)[:, :td]  # noqa: E731
        want += steps.complex_loss_grads(rows(h[sl]), rows(r[sl]), rows(t[sl]),
                                         rows(n[sl]).reshape(-1, cfg.negatives, td))[0]
    assert abs(got - want) <= 1e-4 * abs(want)


def test_sgns_full_size_first_clock_loss(gpu_lib):
    cfg = wl.SGNS
    cen, ctx, neg = (x.numpy() for x in wl.sgns_batch(cfg, 0, 0))
    V = cfg.vocab
    pres = ctx != wl.MISSING
    keys = np.concatenate([cen, V + ctx[pres], V + neg[pres].reshape(-1)])
    ctx32 = np.where(pres, ctx, 0xFFFFFFFF)

    def run(pm, loss):
        pm.sgns_step(0, dev(cen), dev(ctx32.reshape(-1)), dev(neg.reshape(-1)), ctx.shape[1], cfg.negatives,
                     V, cfg.dim, cfg.lr, loss_out=loss)

    got = _first_loss_gpu(gpu_lib, cfg, keys, run, cfg.value_len, cfg.dim)
    want = 0.0
    rows = lambda k: hashgen.init_rows_np(np.asarray(k).reshape(-1), cfg.dim, cfg.dim, cfg.seed, cfg.init_std)  # noqa: E731
    for i in range(cen.size):
        p = pres[i]
        want += steps.sgns_loss_grads(rows([cen[i]])[0], rows(V + ctx[i][p]),
                                      rows(V + neg[i][p]).reshape(int(p.sum()), cfg.negatives, cfg.dim),
                                      np.ones(int(p.sum()), bool))[0]
    assert abs(got - want) <= 1e-4 * abs(want)
