"""GPU parity of the fused training steps (MF, ComplEx, SGNS) against the oracle.

Both sides run the same data-parallel loop (intents signalled `lookahead`
clocks ahead, one step per worker per clock, advance, sync; Fig. 2 pattern)
on the same seeded data.  The GPU computes each sample in fp32, the oracle in
fp64, so the tolerances come from the fp32 arithmetic (u = 2^-24):
  * batch loss of every worker at every clock: relative error <= 1e-4 (the
    stated parity for training losses);
  * one step from identical state (one worker, replicas of the initial
    values): every stored element within 1e-5 of its magnitude bound
    M = |init| + sum |delta| (push summation) plus twice the first-order
    bound B of the fp32 step itself, B computed below from the magnitudes of
    the inputs of each dot product (a forward-error bound: the fp32 error of
    e = v - u.w is at most (d + 2) u (|v| + sum |u_k w_k|), and so on).
    The same check runs at the row widths of the large configurations (MF
    rank 100 + AdaGrad, D = 200; ComplEx 2 x 128 + AdaGrad, D = 512; SGNS
    D = 300), which take the kernels' widest row-group paths;
  * ComplEx's bound B follows the same derivation for the score, the
    logistic coefficients, the weighted tail sum and the head / relation /
    tail gradients (comp_bounds below);
  * after many clocks fp32-vs-fp64 rounding is carried through the dynamics,
    so MF and SGNS trajectories are compared per parameter block at 1e-4 of
    its scale; for ComplEx, whose hottest relation moves by about lr per
    occurrence and compounds that rounding, the oracle's trajectory is
    followed instead (teacher forcing): at several clocks the GPU takes one
    step from the oracle's state, checked per element against B.
"""
import dataclasses

import numpy as np
import pytest
import torch

from oracle import ParameterManagerOracle, driver, steps
from synth import workloads as wl
from synth.hashgen import init_rows_np

pytestmark = pytest.mark.gpu

LOSS_RTOL = 1e-4


def gpu_loop(pm, workers, lookahead, span, nclk, keys_of, work):
    """The application's per-clock loop on the GPU (same order as the oracle's)."""
    for w in range(workers):
        for j in range(lookahead):
            pm.intent(w, keys_of(w, j), j, j + span)
    losses = []
    for c in range(nclk):
        row = []
        for w in range(workers):
            j = c + lookahead
            pm.intent(w, keys_of(w, j), j, j + span)
            row.append(work(w, c))
            pm.advance_clock(w)
        pm.sync()
        losses.append(row)
    pm.wait()
    return [[float(x.item()) for x in r] for r in losses]


def oracle_loop(ref, workers, lookahead, span, nclk, keys_of, work):
    driver.start(ref, workers, lookahead, span, keys_of)
    return [driver.clock(ref, workers, lookahead, span, c, keys_of, work) for c in range(nclk)]


def loss_close(got, want):
    got, want = np.asarray(got), np.asarray(want)
    assert np.all(np.abs(got - want) <= LOSS_RTOL * np.abs(want) + 1e-12), np.max(
        np.abs(got - want) / (np.abs(want) + 1e-30))


def dev(x):
    return torch.as_tensor(np.asarray(x), device="cuda")


def test_tiny_mf_five_epochs(gpu_lib):
    cfg = wl.TINY_MF
    data = wl.tiny_mf_dataset(cfg)
    nclk = wl.tiny_mf_clocks(cfg, data[3])
    init = init_rows_np(np.arange(cfg.num_keys), cfg.value_len, cfg.rank, cfg.seed, cfg.init_std)
    pm = gpu_lib.ParameterManager(cfg.num_keys, cfg.value_len, cfg.workers,
                                  init_values=torch.from_numpy(init).cuda())
    ref = ParameterManagerOracle(cfg.num_keys, cfg.value_len, cfg.workers, init)
    batches = {(w, c): wl.tiny_mf_batch(cfg, data, w, c) for w in range(cfg.workers)
               for c in range(nclk + cfg.lookahead + 1)}

    def keys_np(w, c):
        r, co, _ = batches[(w, c)]
        return np.concatenate([r.numpy(), co.numpy()])

    def work_ref(w, c):
        r, co, v = batches[(w, c)]
        return steps.mf_step(ref, w, r.numpy(), co.numpy(), v.numpy(), cfg.rank, cfg.lr, cfg.adagrad)

    def work_gpu(w, c):
        r, co, v = batches[(w, c)]
        loss = torch.zeros(1, dtype=torch.float64, device="cuda")
        pm.mf_step(w, dev(r), dev(co), v.cuda(), cfg.rank, cfg.adagrad, cfg.lr, loss_out=loss)
        return loss

    want = oracle_loop(ref, cfg.workers, cfg.lookahead, cfg.span, nclk, keys_np, work_ref)
    got = gpu_loop(pm, cfg.workers, cfg.lookahead, cfg.span, nclk, lambda w, c: dev(keys_np(w, c)), work_gpu)
    loss_close(got, want)
    main = pm.read_main(np.arange(cfg.num_keys))
    scale = np.abs(ref.main).max()
    assert np.max(np.abs(main - ref.main)) <= 1e-4 * scale
    # the loss falls on the GPU as well (planted low-rank data)
    per = nclk // cfg.epochs
    ep = [sum(map(sum, got[i * per:(i + 1) * per])) for i in range(cfg.epochs)]
    assert ep[-1] < 0.7 * ep[0]
    pm.close()


def _mf_small_cfg():
    return dataclasses.replace(wl.MF, name="mf_small", rows=2000, cols=300, rank=8, workers=3,
                               batch=700, lookahead=2, zipf_s=1.1, total_cells=10 ** 6)


@pytest.mark.parametrize("relocate,timing", [(False, "start"), (True, "start"), (False, "adaptive"),
                                             (True, "adaptive")])
def test_mf_adagrad_zipf(gpu_lib, relocate, timing):
    cfg = _mf_small_cfg()
    nclk = 6
    init = init_rows_np(np.arange(cfg.num_keys), cfg.value_len, cfg.rank, cfg.seed, cfg.init_std)
    pm = gpu_lib.ParameterManager(cfg.num_keys, cfg.value_len, cfg.workers,
                                  init_values=torch.from_numpy(init).cuda(), relocate=relocate,
                                  action_timing=timing)
    ref = ParameterManagerOracle(cfg.num_keys, cfg.value_len, cfg.workers, init, relocation=relocate,
                                 action_timing=timing)
    batches = {(w, c): wl.mf_batch(cfg, w, c) for w in range(cfg.workers)
               for c in range(nclk + cfg.lookahead + 1)}

    def keys_np(w, c):
        r, co, _ = batches[(w, c)]
        return np.concatenate([r.numpy(), co.numpy()])

    def work_ref(w, c):
        r, co, v = batches[(w, c)]
        return steps.mf_step(ref, w, r.numpy(), co.numpy(), v.numpy(), cfg.rank, cfg.lr, True, cfg.eps)

    def work_gpu(w, c):
        r, co, v = batches[(w, c)]
        loss = torch.zeros(1, dtype=torch.float64, device="cuda")
        pm.mf_step(w, dev(r), dev(co), v.cuda(), cfg.rank, True, cfg.lr, cfg.eps, loss_out=loss)
        return loss

    want = oracle_loop(ref, cfg.workers, cfg.lookahead, cfg.span, nclk, keys_np, work_ref)
    got = gpu_loop(pm, cfg.workers, cfg.lookahead, cfg.span, nclk, lambda w, c: dev(keys_np(w, c)), work_gpu)
    loss_close(got, want)
    main = pm.read_main(np.arange(cfg.num_keys))
    th = slice(0, cfg.rank)
    ac = slice(cfg.rank, 2 * cfg.rank)
    assert np.max(np.abs(main[:, th] - ref.main[:, th])) <= 1e-4 * np.abs(ref.main[:, th]).max()
    assert np.max(np.abs(main[:, ac] - ref.main[:, ac])) <= 1e-4 * np.abs(ref.main[:, ac]).max()
    pm.close()


def _complex_small_cfg():
    return dataclasses.replace(wl.COMPLEX, name="complex_small", entities=400, relations=6, half_dim=8,
                               workers=2, batch=48, negatives=10, lookahead=2, total_triples=10 ** 5)


def test_complex_steps(gpu_lib):
    cfg = _complex_small_cfg()
    nclk = 5
    init = init_rows_np(np.arange(cfg.num_keys), cfg.value_len, cfg.theta_dim, cfg.seed, 0.3)
    pm = gpu_lib.ParameterManager(cfg.num_keys, cfg.value_len, cfg.workers,
                                  init_values=torch.from_numpy(init).cuda())
    ref = ParameterManagerOracle(cfg.num_keys, cfg.value_len, cfg.workers, init)
    batches = {(w, c): wl.complex_batch(cfg, w, c) for w in range(cfg.workers)
               for c in range(nclk + cfg.lookahead + 1)}

    def keys_np(w, c):
        h, r, t, n = batches[(w, c)]
        return np.concatenate([h.numpy(), r.numpy(), t.numpy(), n.numpy().reshape(-1)])

    def work_ref(w, c):
        h, r, t, n = batches[(w, c)]
        return steps.complex_step(ref, w, h.numpy(), r.numpy(), t.numpy(), n.numpy(), cfg.theta_dim,
                                  cfg.lr, cfg.eps)

    def work_gpu(w, c):
        h, r, t, n = batches[(w, c)]
        loss = torch.zeros(1, dtype=torch.float64, device="cuda")
        pm.complex_step(w, dev(h), dev(r), dev(t), dev(n.reshape(-1)), cfg.negatives, cfg.theta_dim,
                        cfg.lr, cfg.eps, loss_out=loss)
        return loss

    # the oracle's trajectory, with the state each clock starts from (worker 0 steps first and
    # reads the values the previous clock's sync left in main)
    driver.start(ref, cfg.workers, cfg.lookahead, cfg.span, keys_np)
    want, states = [], []
    for c in range(nclk):
        states.append(ref.main.copy())
        want.append(driver.clock(ref, cfg.workers, cfg.lookahead, cfg.span, c, keys_np, work_ref))
    got = gpu_loop(pm, cfg.workers, cfg.lookahead, cfg.span, nclk, lambda w, c: dev(keys_np(w, c)), work_gpu)
    loss_close(got, want)
    pm.close()
    # teacher forcing: one step of worker 0's batch from the oracle's state at clocks 1, 3 and 4,
    # every element within the derived bound (a free-running fp32 trajectory compounds rounding
    # through the dominant relation's ~lr-sized AdaGrad steps, so it is compared by its losses)
    for c in (1, 3, nclk - 1):
        h, r, t, ng = (x.numpy() for x in batches[(0, c)])
        complex_one_step_check(gpu_lib, cfg, states[c].astype(np.float32), h, r, t, ng)


def _sgns_small_cfg():
    return dataclasses.replace(wl.SGNS, name="sgns_small", vocab=300, dim=16, workers=2, batch=40,
                               window=2, negatives=3, lookahead=3, total_tokens=2 * 40 * 6)


def test_sgns_steps_with_shard_edges(gpu_lib):
    cfg = _sgns_small_cfg()
    nclk = 6                                  # the shard ends at clock 5: missing right contexts
    init = init_rows_np(np.arange(cfg.num_keys), cfg.value_len, cfg.dim, cfg.seed, 0.3)
    pm = gpu_lib.ParameterManager(cfg.num_keys, cfg.value_len, cfg.workers,
                                  init_values=torch.from_numpy(init).cuda())
    ref = ParameterManagerOracle(cfg.num_keys, cfg.value_len, cfg.workers, init)
    batches = {(w, c): wl.sgns_batch(cfg, w, c) for w in range(cfg.workers)
               for c in range(nclk + cfg.lookahead + 1)}
    V = cfg.vocab

    def keys_np(w, c):
        cen, ctx, neg = (x.numpy() for x in batches[(w, c)])
        pres = ctx != wl.MISSING
        return np.concatenate([cen, V + ctx[pres], V + neg[pres].reshape(-1)])

    def work_ref(w, c):
        cen, ctx, neg = (x.numpy() for x in batches[(w, c)])
        return steps.sgns_step(ref, w, cen, ctx, neg, V, cfg.lr)

    def work_gpu(w, c):
        cen, ctx, neg = batches[(w, c)]
        ctx32 = torch.where(ctx == wl.MISSING, torch.full_like(ctx, 0xFFFFFFFF), ctx)
        loss = torch.zeros(1, dtype=torch.float64, device="cuda")
        pm.sgns_step(w, dev(cen), dev(ctx32.reshape(-1)), dev(neg.reshape(-1)), ctx.shape[1],
                     cfg.negatives, V, cfg.dim, cfg.lr, loss_out=loss)
        return loss

    want = oracle_loop(ref, cfg.workers, cfg.lookahead, cfg.span, nclk, keys_np, work_ref)
    got = gpu_loop(pm, cfg.workers, cfg.lookahead, cfg.span, nclk, lambda w, c: dev(keys_np(w, c)), work_gpu)
    loss_close(got, want)
    main = pm.read_main(np.arange(cfg.num_keys))
    assert np.max(np.abs(main - ref.main)) <= 1e-4 * np.abs(ref.main).max()
    pm.close()


U32 = 2.0 ** -24


def ada_bounds(g, a, dg, lr, eps):
    """First-order fp32 error bounds of the AdaGrad delta row [theta | g*g]."""
    d = -lr * g / np.sqrt(a + g * g + eps)
    sens = lr * (a + eps) / (a + g * g + eps) ** 1.5
    return np.concatenate([sens * dg + 6 * U32 * np.abs(d), 2 * np.abs(g) * dg + dg * dg + U32 * g * g], -1)


def one_step_pair(gpu_lib, K, D, init, keys):
    pm = gpu_lib.ParameterManager(K, D, 1, init_values=torch.from_numpy(init).cuda())
    ref = ParameterManagerOracle(K, D, 1, init)
    for api, k in ((pm, dev(keys)), (ref, keys)):
        api.intent(0, k, 0, 1)             # replicas of the initial values, active now
    return pm, ref


def finish_one_step(pm, ref, K, init, keys_all, deltas_all, bound_all):
    for api in (pm, ref):
        api.advance_clock(0)               # replicas expire: updates merged into main
    main = pm.read_main(np.arange(K))
    M = np.abs(init).astype(np.float64)
    np.add.at(M, keys_all, np.abs(deltas_all))
    B = np.zeros_like(M)
    np.add.at(B, keys_all, bound_all)
    err = np.abs(main.astype(np.float64) - ref.main)
    tol = 1e-5 * M + 2 * B + 1e-30
    assert np.all(err <= tol), float(np.max(err / tol))
    pm.close()


@pytest.mark.parametrize("rank", [8, 100])
def test_mf_one_step_per_element(gpu_lib, rank):
    # rank 100 + AdaGrad is the large MF configuration's row (D = 200)
    cfg = dataclasses.replace(_mf_small_cfg(), rank=rank, batch=700 if rank == 8 else 3000)
    r, co, v = wl.mf_batch(cfg, 0, 0)
    init = init_rows_np(np.arange(cfg.num_keys), cfg.value_len, cfg.rank, cfg.seed, cfg.init_std)
    keys = np.concatenate([r.numpy(), co.numpy()])
    pm, ref = one_step_pair(gpu_lib, cfg.num_keys, cfg.value_len, init, keys)
    steps.mf_step(ref, 0, r.numpy(), co.numpy(), v.numpy(), cfg.rank, cfg.lr, True, cfg.eps)
    pm.mf_step(0, dev(r), dev(co), v.cuda(), cfg.rank, True, cfg.lr, cfg.eps)
    n, d = r.numel(), cfg.rank
    rows = init[keys].astype(np.float64)
    U, Wc = rows[:n, :d], rows[n:, :d]
    vv = v.numpy().astype(np.float64)
    _, gU, gW = steps.mf_loss_grads(U, Wc, vv)
    E = np.abs(vv) + np.sum(np.abs(U * Wc), axis=1)            # magnitude of e's inputs
    dgU = np.abs(Wc) * (d + 3) * U32 * E[:, None]
    dgW = np.abs(U) * (d + 3) * U32 * E[:, None]
    deltas = np.concatenate([steps.delta_rows(gU, rows[:n, d:], cfg.lr, True, cfg.eps),
                             steps.delta_rows(gW, rows[n:, d:], cfg.lr, True, cfg.eps)])
    bound = np.concatenate([ada_bounds(gU, rows[:n, d:], dgU, cfg.lr, cfg.eps),
                            ada_bounds(gW, rows[n:, d:], dgW, cfg.lr, cfg.eps)])
    finish_one_step(pm, ref, cfg.num_keys, init, keys, deltas, bound)


def sigmoid(x):
    return steps.sigmoid(x)


@pytest.mark.parametrize("dim,window,negatives,batch", [(16, 2, 3, 40), (300, 5, 25, 24)])
def test_sgns_one_step_per_element(gpu_lib, dim, window, negatives, batch):
    # dim 300, window 5 and 25 negatives are the large SGNS configuration's
    cfg = dataclasses.replace(_sgns_small_cfg(), dim=dim, window=window, negatives=negatives, batch=batch,
                              vocab=300 if dim == 16 else 3000, total_tokens=2 * batch * 6)
    cen, ctx, neg = (x.numpy() for x in wl.sgns_batch(cfg, 1, 0))   # shard start: missing left contexts
    V, d, lr = cfg.vocab, cfg.dim, cfg.lr
    init = init_rows_np(np.arange(cfg.num_keys), cfg.value_len, cfg.dim, cfg.seed, 0.3)
    pres = ctx != wl.MISSING
    keys = np.concatenate([cen, V + ctx[pres], V + neg[pres].reshape(-1)])
    pm, ref = one_step_pair(gpu_lib, cfg.num_keys, cfg.value_len, init, keys)
    steps.sgns_step(ref, 0, cen, ctx, neg, V, lr)
    ctx32 = np.where(pres, ctx, 0xFFFFFFFF)
    pm.sgns_step(0, dev(cen), dev(ctx32.reshape(-1)), dev(neg.reshape(-1)), ctx.shape[1], cfg.negatives,
                 V, d, lr)
    x0 = init.astype(np.float64)
    kk, dd, bb = [], [], []
    for i in range(cen.size):
        v = x0[cen[i]]
        gv = np.zeros(d)
        bv = np.zeros(d)
        terms = 0
        for j in range(ctx.shape[1]):
            if not pres[i, j]:
                continue
            for q, tok in enumerate([ctx[i, j]] + list(neg[i, j])):
                x = x0[V + tok]
                sc = x @ v
                coef = -sigmoid(-sc) if q == 0 else sigmoid(sc)
                dcoef = 0.25 * (d + 2) * U32 * np.sum(np.abs(x * v)) + 8 * U32 * abs(coef)
                kk.append(V + tok)
                dd.append(-lr * coef * v)
                bb.append(lr * np.abs(v) * dcoef + 2 * U32 * np.abs(lr * coef * v))
                gv += coef * x
                bv += np.abs(x) * dcoef + U32 * np.abs(coef * x)
                terms += 1
        kk.append(cen[i])
        dd.append(-lr * gv)
        bb.append(lr * (bv + (terms + 1) * U32 * np.abs(gv)))
    finish_one_step(pm, ref, cfg.num_keys, init, np.array(kk), np.array(dd), np.array(bb))


def comp_bounds(H, R, T, N, AH, AR, AT, AN, lr, eps):
    """First-order fp32 error bounds of one ComplEx step's delta rows (fp64 inputs).

    H, R, T [n, 2m] theta rows [re | im]; N [n, k, 2m] negative tails; A* the AdaGrad halves.
    With u = 2^-24 and P = (|hr||rr| + |hi||ri|, |hi||rr| + |hr||ri|) (the magnitude of the
    complex product h*r), for a tail x the score phi = sum (h*r)_re x_re + (h*r)_im x_im has
    error <= (2m + 6) u sum P |x|; the coefficient c = -sigma(-phi) or sigma(phi) has error
    <= phi_err / 4 + 8 u |c| (sigma' <= 1/4, expf and the division); the tail gradient c (h*r)
    error <= |dc| P + 4 u |c| P; the weighted tail sum T = sum_j c_j x_j error
    <= E + (k + 4) u Q with E = sum |dc_j| |x_j|, Q = sum |c_j| |x_j|; the head gradient
    (r_re T_re + r_im T_im, r_re T_im - r_im T_re) error <= |r_re| e_re + |r_im| e_im + 3 u
    (|r_re| Q_re + |r_im| Q_im) (and crossed for the imaginary half), the relation gradient
    likewise with h.  Every sum is bounded by its term count, so the bound holds for any
    evaluation order.  Returns keys-order lists (g, dg, acc) per row occurrence:
    head, relation, true tail, negatives."""
    n, td = H.shape
    m = td // 2
    k = N.shape[1]
    hr, hi, rr, ri = H[:, :m], H[:, m:], R[:, :m], R[:, m:]
    Are, Aim = hr * rr - hi * ri, hi * rr + hr * ri
    Pre = np.abs(hr) * np.abs(rr) + np.abs(hi) * np.abs(ri)
    Pim = np.abs(hi) * np.abs(rr) + np.abs(hr) * np.abs(ri)
    X = np.concatenate([T[:, None, :], N], axis=1)                       # [n, 1 + k, 2m]
    phi = np.einsum("nm,njm->nj", Are, X[:, :, :m]) + np.einsum("nm,njm->nj", Aim, X[:, :, m:])
    Mx = np.einsum("nm,njm->nj", Pre, np.abs(X[:, :, :m])) + np.einsum("nm,njm->nj", Pim, np.abs(X[:, :, m:]))
    dphi = (2 * m + 6) * U32 * Mx
    c = np.concatenate([-sigmoid(-phi[:, :1]), sigmoid(phi[:, 1:])], axis=1)
    dc = 0.25 * dphi + 8 * U32 * np.abs(c)
    P = np.concatenate([Pre, Pim], axis=1)                               # [n, 2m]
    A = np.concatenate([Are, Aim], axis=1)
    gX = c[:, :, None] * A[:, None, :]
    dgX = dc[:, :, None] * P[:, None, :] + 4 * U32 * np.abs(c)[:, :, None] * P[:, None, :]
    Tt = np.einsum("nj,njd->nd", c, X)
    Q = np.einsum("nj,njd->nd", np.abs(c), np.abs(X))
    E = np.einsum("nj,njd->nd", dc, np.abs(X)) + (k + 4) * U32 * Q
    Tre, Tim = Tt[:, :m], Tt[:, m:]
    Er, Ei, Qr, Qi = E[:, :m], E[:, m:], Q[:, :m], Q[:, m:]

    def lin(a, b):   # gradient (a T_re + b T_im, a T_im - b T_re) and its bound
        g = np.concatenate([a * Tre + b * Tim, a * Tim - b * Tre], axis=1)
        aa, bb = np.abs(a), np.abs(b)
        dg = np.concatenate([aa * Er + bb * Ei + 3 * U32 * (aa * Qr + bb * Qi),
                             aa * Ei + bb * Er + 3 * U32 * (aa * Qi + bb * Qr)], axis=1)
        return g, dg

    gH, dgH = lin(rr, ri)
    gR, dgR = lin(hr, hi)
    out_g = [gH, gR, gX[:, 0], gX[:, 1:].reshape(n * k, td)]
    out_dg = [dgH, dgR, dgX[:, 0], dgX[:, 1:].reshape(n * k, td)]
    out_a = [AH, AR, AT, AN.reshape(n * k, td)]
    g = np.concatenate(out_g)
    dg = np.concatenate(out_dg)
    a = np.concatenate(out_a)
    deltas = steps.delta_rows(g, a, lr, True, eps)
    return deltas, ada_bounds(g, a, dg, lr, eps)


def complex_one_step_check(gpu_lib, cfg, init, h, r, t, ng):
    """One ComplEx step from identical state (init), one worker: loss within 1e-4 and every
    stored element within 1e-5 M + 2 B (comp_bounds)."""
    keys = np.concatenate([h, r, t, ng.reshape(-1)])
    pm, ref = one_step_pair(gpu_lib, cfg.num_keys, cfg.value_len, init, keys)
    want = steps.complex_step(ref, 0, h, r, t, ng, cfg.theta_dim, cfg.lr, cfg.eps)
    loss = torch.zeros(1, dtype=torch.float64, device="cuda")
    pm.complex_step(0, dev(h), dev(r), dev(t), dev(ng.reshape(-1)), cfg.negatives, cfg.theta_dim, cfg.lr,
                    cfg.eps, loss_out=loss)
    pm.wait()
    assert abs(float(loss.item()) - want) <= LOSS_RTOL * abs(want)
    td = cfg.theta_dim
    x0 = init.astype(np.float64)
    n = h.size
    th = lambda kk: x0[kk, :td]     # noqa: E731
    ac = lambda kk: x0[kk, td:]     # noqa: E731
    deltas, bound = comp_bounds(th(h), th(r), th(t), th(ng.reshape(-1)).reshape(n, -1, td),
                                ac(h), ac(r), ac(t), ac(ng.reshape(-1)).reshape(n, -1, td), cfg.lr, cfg.eps)
    finish_one_step(pm, ref, cfg.num_keys, init, keys, deltas, bound)


@pytest.mark.parametrize("half_dim,negatives,batch", [(8, 10, 48), (128, 100, 40)])
def test_complex_one_step_per_element(gpu_lib, half_dim, negatives, batch):
    """One ComplEx step from identical state; half_dim 128 with 100 negatives is the large
    ComplEx configuration's row (D = 512)."""
    cfg = dataclasses.replace(_complex_small_cfg(), half_dim=half_dim, negatives=negatives, batch=batch,
                              entities=400 if half_dim == 8 else 3000)
    h, r, t, ng = (x.numpy() for x in wl.complex_batch(cfg, 0, 0))
    init = init_rows_np(np.arange(cfg.num_keys), cfg.value_len, cfg.theta_dim, cfg.seed, 0.3)
    # a non-zero accumulator half, as after some training, so both AdaGrad inputs matter
    init[:, cfg.theta_dim:] = np.abs(init_rows_np(np.arange(cfg.num_keys), cfg.value_len, cfg.theta_dim,
                                                  cfg.seed + 5, 0.3))[:, :cfg.theta_dim]
    complex_one_step_check(gpu_lib, cfg, init, h, r, t, ng)
