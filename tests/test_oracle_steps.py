"""Pins of the oracle's training steps (App. C tasks) against independent computations.

* gradients against fp64 central finite differences of the loss;
* the ComplEx score against Python complex arithmetic Re(sum h r conj(t)),
  and its DistMult special case (all-real rows);
* closed forms: zero vectors give softplus(0) = log 2 per score; the AdaGrad
  delta on hand numbers;
* a single worker with sync every clock reproduces textbook mini-batch SGD, and with
  AdaGrad a textbook mini-batch AdaGrad loop (the large MF configuration's path);
* keys repeated inside one batch take one AdaGrad step per occurrence (MF on hand numbers,
  ComplEx against per-occurrence finite differences), told apart from summing first;
* MF loss falls on the tiny planted-rank workload.

Planted mistakes in a scratch copy of the oracle's MF step were caught: swapping the
row and column accumulators fails the textbook AdaGrad loop; dropping the g*g half of the
delta row, or summing a key's gradients before one AdaGrad step, fails both MF pins.
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


# ---------------------------------------------------------------------------
# AdaGrad (App. C: "SGD with AdaGrad"): the MF branch and repeated keys
# ---------------------------------------------------------------------------

def _textbook_minibatch_adagrad_mf(theta, acc, rank, batches, lr, eps):
    """Mini-batch AdaGrad on 1/2 (v - u.w)^2 with a single store (no parameter manager).

    theta [K, rank] factors, acc [K, rank] squared-gradient accumulators, fp64.
    Every cell of a batch reads the store as it was at the start of the batch;
    each occurrence of a factor row in a cell takes its own AdaGrad step
    against the accumulator read at the start of the batch:
        a_occ = acc[k] + g^2,  theta[k] -= lr g / sqrt(a_occ + eps),  acc[k] += g^2.
    """
    theta = theta.astype(np.float64).copy()
    acc = acc.astype(np.float64).copy()
    for rows, cols, vals in batches:
        th0, ac0 = theta.copy(), acc.copy()
        for i in range(len(rows)):
            u, w = int(rows[i]), int(cols[i])
            e = float(vals[i]) - float(th0[u] @ th0[w])
            for k, g in ((u, -e * th0[w]), (w, -e * th0[u])):
                theta[k] -= lr * g / np.sqrt(ac0[k] + g * g + eps)
                acc[k] += g * g
    return theta, acc


def test_single_worker_adagrad_equals_textbook_minibatch_adagrad():
    """The MF step with AdaGrad (the large MF configuration's path), one worker, sync every clock:
    the manager's result equals a plain AdaGrad loop over the same batches.  Swapping the
    accumulators of the row and column factor (or dropping the g*g half of the delta row) moves
    the result by O(1) relative and fails this test (checked on a scratch copy of the oracle)."""
    import dataclasses
    cfg = dataclasses.replace(wl.TINY_MF, workers=1, epochs=1, adagrad=True, rank=8, lr=0.05)
    data = wl.tiny_mf_dataset(cfg)
    nclk = 25
    init = init_rows_np(np.arange(cfg.num_keys), cfg.value_len, cfg.rank, cfg.seed, cfg.init_std)
    assert init.shape[1] == 2 * cfg.rank and not init[:, cfg.rank:].any()   # accumulators start at 0
    # a non-zero starting accumulator so that a swapped or misplaced accumulator cannot go unnoticed
    rng = np.random.default_rng(21)
    init[:, cfg.rank:] = rng.uniform(0.01, 0.5, size=(cfg.num_keys, cfg.rank)).astype(np.float32)
    pm = ParameterManagerOracle(cfg.num_keys, cfg.value_len, 1, init)
    batches = [tuple(x.numpy() for x in wl.tiny_mf_batch(cfg, data, 0, c)) for c in range(nclk + 3)]

    def keys_of(w, c):
        return np.concatenate(batches[c][:2])

    def work(w, c):
        r, co, v = batches[c]
        return steps.mf_step(pm, w, r, co, v, cfg.rank, cfg.lr, True, cfg.eps)

    driver.start(pm, 1, cfg.lookahead, cfg.span, keys_of)
    for c in range(nclk):
        driver.clock(pm, 1, cfg.lookahead, cfg.span, c, keys_of, work)
    th, ac = _textbook_minibatch_adagrad_mf(init[:, :cfg.rank], init[:, cfg.rank:], cfg.rank,
                                            [batches[c] for c in range(nclk)], cfg.lr, cfg.eps)
    # the manager stores fp32 after every clock; the textbook loop keeps fp64
    assert np.allclose(pm.main[:, :cfg.rank], th, rtol=1e-5, atol=1e-6)
    assert np.allclose(pm.main[:, cfg.rank:], ac, rtol=1e-5, atol=1e-6)
    assert not np.allclose(pm.main[:, :cfg.rank], init[:, :cfg.rank], atol=1e-3)


def test_mf_adagrad_repeated_key_takes_one_step_per_occurrence():
    """Hand numbers, rank 1, eps 0, lr 1/2: row u = 1 meets columns w1 = 2 and w2 = -1 (values 0).
    e1 = -2, e2 = 1; the row's gradients per occurrence are 4 and 1, the columns' 2 and -1.
    Per occurrence: theta_u += -1/2 (4/sqrt(16) + 1/sqrt(1)) = -1, a_u += 16 + 1 = 17.
    (Summing first would give theta_u += -1/2 * 5/sqrt(25) = -1/2 and a_u += 25.)"""
    init = np.array([[1.0, 0.0], [2.0, 0.0], [-1.0, 0.0]], np.float32)   # [theta | a] of u, w1, w2
    pm = ParameterManagerOracle(3, 2, 1, init)                          # no intents: pushes go to main
    loss = steps.mf_step(pm, 0, np.array([0, 0]), np.array([1, 2]), np.array([0.0, 0.0], np.float32),
                         1, 0.5, True, 0.0)
    assert loss == 2.5
    assert np.array_equal(pm.main, np.array([[0.0, 17.0], [1.5, 4.0], [-0.5, 1.0]], np.float32))


def test_complex_adagrad_repeated_keys_take_one_step_per_occurrence():
    """ComplEx with keys repeated inside one batch (a relation in both triples, an entity that is the
    head of one triple and a negative tail of the other): every row occurrence takes its own AdaGrad
    step with its own gradient, which is found here by fp64 finite differences of the batch loss with
    respect to that occurrence alone (each occurrence made a variable of its own)."""
    m, K = 2, 8
    td = 2 * m
    rng = np.random.default_rng(41)
    init = np.zeros((K, 2 * td), np.float32)
    init[:, :td] = rng.normal(0, 0.7, size=(K, td))
    init[:, td:] = rng.uniform(0.05, 0.5, size=(K, td))
    heads, rels, tails = [0, 1], [6, 6], [2, 3]
    negs = [[4, 1], [0, 4]]                      # entity 1: head of triple 1 and a negative of triple 0
    lr, eps = 0.1, 1e-8
    pm = ParameterManagerOracle(K, 2 * td, 1, init)
    steps.complex_step(pm, 0, heads, rels, tails, negs, td, lr, eps)

    occ = heads + rels + tails + [k for row in negs for k in row]      # the step's row occurrences
    x0 = init[occ, :td].astype(np.float64)                             # one variable per occurrence
    n, k = len(heads), len(negs[0])

    def loss_of(x):
        total = 0.0
        for i in range(n):
            h, r, t = x[i], x[n + i], x[2 * n + i]
            z = lambda a, b, c: sum(complex(a[q], a[m + q]) * complex(b[q], b[m + q]) *  # noqa: E731
                                    complex(c[q], -c[m + q]) for q in range(m)).real
            total += math.log1p(math.exp(-z(h, r, t)))
            for j in range(k):
                total += math.log1p(math.exp(z(h, r, x[3 * n + i * k + j])))
        return total

    g = fd_grad(loss_of, x0)
    acc0 = init[occ, td:].astype(np.float64)
    want = init.astype(np.float64).copy()
    for o, key in enumerate(occ):
        want[key, :td] += -lr * g[o] / np.sqrt(acc0[o] + g[o] * g[o] + eps)
        want[key, td:] += g[o] * g[o]
    assert np.allclose(pm.main, want, rtol=1e-5, atol=1e-7)
    # the alternative reading (sum a key's gradients, then one AdaGrad step) is told apart
    alt = init.astype(np.float64).copy()
    for key in set(occ):
        gs = sum(g[o] for o in range(len(occ)) if occ[o] == key)
        alt[key, :td] += -lr * gs / np.sqrt(init[key, td:] + gs * gs + eps)
        alt[key, td:] += gs * gs
    assert not np.allclose(alt, want, rtol=1e-5, atol=1e-7)
