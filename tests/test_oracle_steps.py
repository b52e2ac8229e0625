"""Pins of the oracle's training steps (App. C tasks) against independent computations.

* gradients against fp64 central finite differences of the loss;
* the ComplEx score against Python complex arithmetic Re(sum h r conj(t)),
  and its DistMult special case (all-real rows);
* closed forms: zero vectors give softplus(0) = log 2 per score; the AdaGrad
  delta on hand numbers;
* a single worker with sync every clock reproduces textbook mini-batch SGD;
* MF loss falls on the tiny planted-rank workload.
"""
import math

import numpy as np
import pytest

from oracle import ParameterManagerOracle, driver, steps
from synth import workloads as wl
from synth.hashgen import init_rows_np


def fd_grad(f, x, h=1e-6):
    g = np.zeros_like(x)
    it = np.nditer(x, flags=["multi_index"])
    for _ in it:
        i = it.multi_index
        xp = x.copy()
        xm = x.copy()
        xp[i] += h
        xm[i] -= h
        g[i] = (f(xp) - f(xm)) / (2 * h)
    return g


def test_mf_gradients_finite_differences():
    rng = np.random.default_rng(0)
    U = rng.normal(size=(3, 5))
    Wc = rng.normal(size=(3, 5))
    v = rng.normal(size=3)
    loss, gU, gW = steps.mf_loss_grads(U, Wc, v)
    assert np.isclose(loss, 0.5 * sum((v[i] - U[i] @ Wc[i]) ** 2 for i in range(3)))
    assert np.allclose(gU, fd_grad(lambda x: steps.mf_loss_grads(x, Wc, v)[0], U), atol=1e-6)
    assert np.allclose(gW, fd_grad(lambda x: steps.mf_loss_grads(U, x, v)[0], Wc), atol=1e-6)


def test_complex_score_matches_complex_arithmetic():
    rng = np.random.default_rng(1)
    m = 4
    h, r, t = (rng.normal(size=2 * m) for _ in range(3))
    z = sum(complex(h[k], h[m + k]) * complex(r[k], r[m + k]) * complex(t[k], -t[m + k])
            for k in range(m))
    assert math.isclose(steps.complex_score(h, r, t), z.real, rel_tol=1e-12, abs_tol=1e-12)
    # all-real rows reduce ComplEx to DistMult: sum_k h_k r_k t_k
    hr, rr, tr = (np.concatenate([x[:m], np.zeros(m)]) for x in (h, r, t))
    assert math.isclose(steps.complex_score(hr, rr, tr), float(np.sum(h[:m] * r[:m] * t[:m])),
                        rel_tol=1e-12)
    # antisymmetry of ComplEx in (h, t) for purely imaginary relations
    ri = np.concatenate([np.zeros(m), r[m:]])
    assert math.isclose(steps.complex_score(h, ri, t), -steps.complex_score(t, ri, h),
                        rel_tol=1e-12, abs_tol=1e-12)


def test_complex_gradients_finite_differences():
    rng = np.random.default_rng(2)
    n, k, d = 2, 3, 6
    H, R, T = (rng.normal(size=(n, d)) for _ in range(3))
    N = rng.normal(size=(n, k, d))
    loss, gH, gR, gT, gN = steps.complex_loss_grads(H, R, T, N)
    f = steps.complex_loss_grads
    assert np.allclose(gH, fd_grad(lambda x: f(x, R, T, N)[0], H), atol=1e-6)
    assert np.allclose(gR, fd_grad(lambda x: f(H, x, T, N)[0], R), atol=1e-6)
    assert np.allclose(gT, fd_grad(lambda x: f(H, R, x, N)[0], T), atol=1e-6)
    assert np.allclose(gN, fd_grad(lambda x: f(H, R, T, x)[0], N), atol=1e-6)
    # loss against logistic loss written with math.log / math.exp
    want = 0.0
    for i in range(n):
        want += math.log(1 + math.exp(-steps.complex_score(H[i], R[i], T[i])))
        for j in range(k):
            want += math.log(1 + math.exp(steps.complex_score(H[i], R[i], N[i, j])))
    assert math.isclose(loss, want, rel_tol=1e-12)


def test_sgns_gradients_and_closed_form():
    rng = np.random.default_rng(3)
    c, k, d = 3, 4, 5
    v = rng.normal(size=d)
    Uc = rng.normal(size=(c, d))
    Un = rng.normal(size=(c, k, d))
    pres = np.array([True, False, True])
    f = steps.sgns_loss_grads
    loss, gv, gc, gn = f(v, Uc, Un, pres)
    assert np.allclose(gv, fd_grad(lambda x: f(x, Uc, Un, pres)[0], v), atol=1e-6)
    assert np.allclose(gc, fd_grad(lambda x: f(v, x, Un, pres)[0], Uc), atol=1e-6)
    assert np.allclose(gn, fd_grad(lambda x: f(v, Uc, x, pres)[0], Un), atol=1e-6)
    want = 0.0
    for j in range(c):
        if pres[j]:
            want += -math.log(1 / (1 + math.exp(-Uc[j] @ v)))
            want += sum(-math.log(1 / (1 + math.exp(Un[j, q] @ v))) for q in range(k))
    assert math.isclose(loss, want, rel_tol=1e-12)
    # zero vectors: every score is 0 and costs log 2
    z = f(np.zeros(d), np.zeros((c, d)), np.zeros((c, k, d)), np.ones(c, bool))[0]
    assert math.isclose(z, c * (1 + k) * math.log(2.0), rel_tol=1e-15)


def test_stable_softplus_and_sigmoid():
    for x in (-800.0, -30.0, -1.5, 0.0, 2.0, 40.0, 800.0):
        sp = steps.softplus(x)
        ref = x + math.log1p(math.exp(-x)) if x > 0 else math.log1p(math.exp(x))
        assert math.isclose(sp, ref, rel_tol=1e-14, abs_tol=1e-300)
        s = steps.sigmoid(x)
        ref = 1 / (1 + math.exp(-x)) if x > -700 else 0.0
        assert math.isclose(s, ref, rel_tol=1e-14, abs_tol=1e-300)


def test_adagrad_delta_hand_numbers():
    # g = 2, a = 5, lr = 0.1: a' = 9, delta theta = -0.1 * 2 / 3, delta a = 4
    d = steps.delta_rows(np.array([[2.0]]), np.array([[5.0]]), 0.1, True, 0.0)
    assert np.allclose(d, [[-0.2 / 3.0, 4.0]], rtol=1e-15)
    d = steps.delta_rows(np.array([[2.0, -1.0]]), None, 0.5, False, 0.0)
    assert np.allclose(d, [[-1.0, 0.5]])


def _textbook_minibatch_sgd(theta, batches, lr):
    """Plain single-store mini-batch SGD on 1/2 (v - u.w)^2 (no parameter manager)."""
    theta = theta.astype(np.float64)
    for rows, cols, vals in batches:
        U, Wc = theta[rows], theta[cols]
        e = vals - np.einsum("ij,ij->i", U, Wc)
        upd = np.zeros_like(theta)
        np.add.at(upd, rows, lr * e[:, None] * Wc)
        np.add.at(upd, cols, lr * e[:, None] * U)
        theta = theta + upd
    return theta


def _run_tiny_mf(cfg, data, epochs_clocks=None):
    init = init_rows_np(np.arange(cfg.num_keys), cfg.value_len, cfg.rank, cfg.seed, cfg.init_std)
    pm = ParameterManagerOracle(cfg.num_keys, cfg.value_len, cfg.workers, init)
    nclk = wl.tiny_mf_clocks(cfg, data[3]) if epochs_clocks is None else epochs_clocks

    def keys_of(w, c):
        r, co, _ = wl.tiny_mf_batch(cfg, data, w, c)
        return np.concatenate([r.numpy(), co.numpy()])

    def work(w, c):
        r, co, v = wl.tiny_mf_batch(cfg, data, w, c)
        return steps.mf_step(pm, w, r.numpy(), co.numpy(), v.numpy(), cfg.rank, cfg.lr, cfg.adagrad)

    driver.start(pm, cfg.workers, cfg.lookahead, cfg.span, keys_of)
    losses = [sum(driver.clock(pm, cfg.workers, cfg.lookahead, cfg.span, c, keys_of, work))
              for c in range(nclk)]
    return pm, init, losses, nclk


def test_single_worker_equals_textbook_minibatch_sgd():
    import dataclasses
    cfg = dataclasses.replace(wl.TINY_MF, workers=1, epochs=1)
    data = wl.tiny_mf_dataset(cfg)
    nclk = 30
    pm, init, _, _ = _run_tiny_mf(cfg, data, nclk)
    pm.sync()
    batches = []
    for c in range(nclk):
        r, co, v = wl.tiny_mf_batch(cfg, data, 0, c)
        batches.append((r.numpy(), co.numpy(), v.numpy().astype(np.float64)))
    want = _textbook_minibatch_sgd(init, batches, cfg.lr)
    # the manager stores fp32 after every clock; the textbook loop keeps fp64
    assert np.allclose(pm.main, want, rtol=2e-6, atol=2e-7)
    assert not np.allclose(pm.main, init, atol=1e-3)


def test_mf_loss_falls_on_planted_low_rank_data():
    cfg = wl.TINY_MF
    data = wl.tiny_mf_dataset(cfg)
    _, _, losses, nclk = _run_tiny_mf(cfg, data)
    per = nclk // cfg.epochs
    epoch = [sum(losses[i * per:(i + 1) * per]) for i in range(cfg.epochs)]
    assert all(b < a for a, b in zip(epoch, epoch[1:])), epoch
    assert epoch[-1] < 0.7 * epoch[0], epoch


def _complex_batch_loss_via_complex_numbers(rows, heads, rels, tails, negs, m):
    """Batch loss from stored theta rows, written with Python complex numbers."""
    def c(row):
        return [complex(row[k], row[m + k]) for k in range(m)]

    def phi(h, r, t):
        return sum(a * b * z.conjugate() for a, b, z in zip(c(h), c(r), c(t))).real

    total = 0.0
    for i in range(len(heads)):
        h, r, t = rows[heads[i]], rows[rels[i]], rows[tails[i]]
        total += math.log1p(math.exp(-phi(h, r, t)))
        for nk in negs[i]:
            total += math.log1p(math.exp(phi(h, r, rows[nk])))
    return total


def test_complex_step_pushes_adagrad_deltas_of_the_batch_gradient():
    m, K = 3, 10
    td = 2 * m
    rng = np.random.default_rng(4)
    init = np.zeros((K, 2 * td), np.float32)
    init[:, :td] = rng.normal(0, 0.5, size=(K, td))
    init[:, td:] = rng.uniform(0.1, 1.0, size=(K, td))      # some accumulated AdaGrad state
    pm = ParameterManagerOracle(K, 2 * td, 1, init)          # no intents: pushes go to main
    heads, rels, tails, negs = [0, 1], [8, 9], [2, 3], [[4, 5], [6, 7]]
    lr, eps = 0.1, 1e-8
    loss = steps.complex_step(pm, 0, heads, rels, tails, negs, td, lr, eps)
    theta = init[:, :td].astype(np.float64)
    g = fd_grad(lambda x: _complex_batch_loss_via_complex_numbers(x, heads, rels, tails, negs, m), theta)
    assert math.isclose(loss, _complex_batch_loss_via_complex_numbers(theta, heads, rels, tails, negs, m),
                        rel_tol=1e-7)
    a_new = init[:, td:].astype(np.float64) + g * g
    want_theta = init[:, :td] - lr * g / np.sqrt(a_new + eps)
    assert np.allclose(pm.main[:, :td], want_theta, rtol=1e-5, atol=1e-7)
    assert np.allclose(pm.main[:, td:], a_new, rtol=1e-5, atol=1e-7)


def test_sgns_step_pushes_sgd_deltas_of_the_batch_gradient():
    V, d, k = 6, 4, 2
    rng = np.random.default_rng(6)
    init = rng.normal(0, 0.5, size=(2 * V, d)).astype(np.float32)
    pm = ParameterManagerOracle(2 * V, d, 1, init)
    centres = [0, 3]
    contexts = [[1, -1], [2, 4]]                 # one missing context slot
    negs = [[[5, 2], [0, 0]], [[1, 1], [3, 5]]]
    lr = 0.05

    def batch_loss(x):
        tot = 0.0
        for i, cidx in enumerate(centres):
            for j, o in enumerate(contexts[i]):
                if o < 0:
                    continue
                tot -= math.log(1 / (1 + math.exp(-(x[V + o] @ x[cidx]))))
                for nk in negs[i][j]:
                    tot -= math.log(1 / (1 + math.exp(x[V + nk] @ x[cidx])))
        return tot

    loss = steps.sgns_step(pm, 0, centres, contexts, negs, V, lr)
    x0 = init.astype(np.float64)
    assert math.isclose(loss, batch_loss(x0), rel_tol=1e-9)
    g = fd_grad(batch_loss, x0)
    assert np.allclose(pm.main, x0 - lr * g, rtol=1e-5, atol=1e-7)
