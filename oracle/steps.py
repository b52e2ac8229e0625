"""Oracle of the three training steps that consume pulled rows (App. C).

TEST INFRASTRUCTURE ONLY (see oracle/__init__.py).

A step of worker w on one batch pulls every row the batch touches, computes
each sample's loss and gradients from those pulled values (later samples of
the batch do not see earlier samples' updates), turns each gradient into a
delta row, and pushes all delta rows once.  Everything is fp64; delta rows
are rounded to fp32 when pushed.

Optimiser (App. C: "SGD with AdaGrad" for every task).  With AdaGrad the
value row is [theta | a]: a is the accumulator of squared gradients.  For a
gradient g of one row occurrence, a' = a + g*g and the delta row is
[-lr * g / sqrt(a' + eps) | g*g], so push and sync stay purely additive.
Without AdaGrad the delta row is -lr * g.

Losses (the paper names the models, not the formulas):
  MF        1/2 (v - u.w)^2 for a cell (row u, column w, value v)
  ComplEx   phi(h, r, t) = Re(sum_k h_k r_k conj(t_k)) with rows stored as
            [re | im]; loss softplus(-y phi), y = +1 for the true tail and
            -1 for each negative tail (Trouillon et al., ComplEx)
  SGNS      softplus(-u_o.v_c) + sum_n softplus(u_n.v_c) per (centre, context)
            pair; v = input vectors (keys [0, V)), u = output vectors (keys
            [V, 2V)) (Mikolov et al., skip-gram with negative sampling)
"""
import numpy as np

MISSING = -1


def softplus(x):
    x = np.asarray(x, dtype=np.float64)
    return np.log1p(np.exp(-np.abs(x))) + np.maximum(x, 0.0)


def sigmoid(x):
    x = np.asarray(x, dtype=np.float64)
    return np.where(x >= 0, 1.0 / (1.0 + np.exp(-np.abs(x))), np.exp(-np.abs(x)) / (1.0 + np.exp(-np.abs(x))))


def delta_rows(theta_grad, acc, lr, adagrad, eps):
    """Delta rows for gradients of row occurrences (fp64 in, fp64 out)."""
    g = np.asarray(theta_grad, dtype=np.float64)
    if not adagrad:
        return -lr * g
    a_new = np.asarray(acc, dtype=np.float64) + g * g
    return np.concatenate([-lr * g / np.sqrt(a_new + eps), g * g], axis=-1)


# ---------------------------------------------------------------------------
# matrix factorisation
# ---------------------------------------------------------------------------

def mf_loss_grads(U, Wc, vals):
    """Loss and gradients of cells; U, Wc: [n, r] fp64, vals [n]."""
    U = np.asarray(U, dtype=np.float64)
    Wc = np.asarray(Wc, dtype=np.float64)
    e = np.asarray(vals, dtype=np.float64) - np.sum(U * Wc, axis=1)
    loss = 0.5 * np.sum(e * e)
    gU = -e[:, None] * Wc
    gW = -e[:, None] * U
    return loss, gU, gW


def mf_step(pm, w, row_keys, col_keys, vals, rank, lr, adagrad, eps=1e-8):
    n = len(row_keys)
    if n == 0:
        return 0.0
    keys = np.concatenate([np.asarray(row_keys), np.asarray(col_keys)]).astype(np.int64)
    rows = pm.pull(w, keys).astype(np.float64)
    U, Wc = rows[:n, :rank], rows[n:, :rank]
    loss, gU, gW = mf_loss_grads(U, Wc, vals)
    acc_u = rows[:n, rank:] if adagrad else None
    acc_w = rows[n:, rank:] if adagrad else None
    d = np.concatenate([delta_rows(gU, acc_u, lr, adagrad, eps),
                        delta_rows(gW, acc_w, lr, adagrad, eps)])
    pm.push(w, keys, d.astype(np.float32))
    return float(loss)


# ---------------------------------------------------------------------------
# ComplEx
# ---------------------------------------------------------------------------

def complex_score(h, r, t):
    """phi for theta rows [re | im] (last axis), broadcasting over leading axes."""
    h = np.asarray(h, dtype=np.float64)
    r = np.asarray(r, dtype=np.float64)
    t = np.asarray(t, dtype=np.float64)
    m = h.shape[-1] // 2
    hr, hi = h[..., :m], h[..., m:]
    rr, ri = r[..., :m], r[..., m:]
    tr, ti = t[..., :m], t[..., m:]
    return np.sum(hr * rr * tr + hi * rr * ti + hr * ri * ti - hi * ri * tr, axis=-1)


def complex_score_grads(h, r, t):
    """d phi / d h, d phi / d r, d phi / d t (rows [re | im])."""
    m = h.shape[-1] // 2
    hr, hi = h[..., :m], h[..., m:]
    rr, ri = r[..., :m], r[..., m:]
    tr, ti = t[..., :m], t[..., m:]
    dh = np.concatenate([rr * tr + ri * ti, rr * ti - ri * tr], axis=-1)
    dr = np.concatenate([hr * tr + hi * ti, hr * ti - hi * tr], axis=-1)
    dt = np.concatenate([hr * rr - hi * ri, hi * rr + hr * ri], axis=-1)
    return dh, dr, dt


def complex_loss_grads(H, R, T, N):
    """One batch: H, R, T [n, 2m]; N [n, k, 2m] negative tails.

    Returns loss and gradients gH, gR, gT [n, 2m], gN [n, k, 2m].
    """
    H = np.asarray(H, dtype=np.float64)
    R = np.asarray(R, dtype=np.float64)
    T = np.asarray(T, dtype=np.float64)
    N = np.asarray(N, dtype=np.float64)
    pos = complex_score(H, R, T)                          # [n]
    neg = complex_score(H[:, None, :], R[:, None, :], N)  # [n, k]
    loss = np.sum(softplus(-pos)) + np.sum(softplus(neg))
    cp = -sigmoid(-pos)                                   # d softplus(-x) / dx
    cn = sigmoid(neg)                                     # d softplus(x) / dx
    dh_p, dr_p, dt_p = complex_score_grads(H, R, T)
    dh_n, dr_n, dt_n = complex_score_grads(H[:, None, :], R[:, None, :], N)
    gH = cp[:, None] * dh_p + np.sum(cn[:, :, None] * dh_n, axis=1)
    gR = cp[:, None] * dr_p + np.sum(cn[:, :, None] * dr_n, axis=1)
    gT = cp[:, None] * dt_p
    gN = cn[:, :, None] * dt_n
    return loss, gH, gR, gT, gN


def complex_step(pm, w, heads, rels, tails, negs, theta_dim, lr, eps=1e-8):
    heads = np.asarray(heads, dtype=np.int64)
    n = heads.size
    if n == 0:
        return 0.0
    negs = np.asarray(negs, dtype=np.int64).reshape(n, -1)
    k = negs.shape[1]
    keys = np.concatenate([heads, np.asarray(rels, np.int64), np.asarray(tails, np.int64),
                           negs.reshape(-1)])
    rows = pm.pull(w, keys).astype(np.float64)
    H, R, T = rows[:n], rows[n:2 * n], rows[2 * n:3 * n]
    Nr = rows[3 * n:].reshape(n, k, -1)
    td = theta_dim
    loss, gH, gR, gT, gN = complex_loss_grads(H[:, :td], R[:, :td], T[:, :td], Nr[:, :, :td])
    d = np.concatenate([
        delta_rows(gH, H[:, td:], lr, True, eps),
        delta_rows(gR, R[:, td:], lr, True, eps),
        delta_rows(gT, T[:, td:], lr, True, eps),
        delta_rows(gN.reshape(n * k, td), Nr[:, :, td:].reshape(n * k, td), lr, True, eps),
    ])
    pm.push(w, keys, d.astype(np.float32))
    return float(loss)


# ---------------------------------------------------------------------------
# skip-gram with negative sampling
# ---------------------------------------------------------------------------

def sgns_loss_grads(v, U_ctx, U_neg, present):
    """One centre: v [d]; U_ctx [c, d] context outputs; U_neg [c, k, d]; present [c] bool.

    Returns loss, g_v [d], g_ctx [c, d], g_neg [c, k, d] (zero where absent).
    """
    v = np.asarray(v, dtype=np.float64)
    U_ctx = np.asarray(U_ctx, dtype=np.float64)
    U_neg = np.asarray(U_neg, dtype=np.float64)
    pres = np.asarray(present, dtype=bool)
    sp = U_ctx @ v                                  # [c]
    sn = U_neg @ v                                  # [c, k]
    loss = np.sum(np.where(pres, softplus(-sp), 0.0)) + np.sum(np.where(pres[:, None], softplus(sn), 0.0))
    cp = np.where(pres, -sigmoid(-sp), 0.0)
    cn = np.where(pres[:, None], sigmoid(sn), 0.0)
    g_v = cp @ U_ctx + np.einsum("ck,ckd->d", cn, U_neg)
    g_ctx = cp[:, None] * v[None, :]
    g_neg = cn[:, :, None] * v[None, None, :]
    return loss, g_v, g_ctx, g_neg


def sgns_step(pm, w, centres, contexts, negs, vocab, lr):
    """Plain-SGD skip-gram step; keys: centre c -> c, output token o -> vocab + o."""
    centres = np.asarray(centres, dtype=np.int64)
    contexts = np.asarray(contexts, dtype=np.int64)
    negs = np.asarray(negs, dtype=np.int64)
    n = centres.size
    if n == 0:
        return 0.0
    keys, deltas = [], []
    loss = 0.0
    for i in range(n):
        pres = contexts[i] != MISSING
        ctx_keys = vocab + contexts[i][pres]
        neg_keys = vocab + negs[i][pres]                      # [c', k]
        my_keys = np.concatenate([[centres[i]], ctx_keys, neg_keys.reshape(-1)])
        rows = pm.pull(w, my_keys).astype(np.float64)
        c = ctx_keys.size
        v = rows[0]
        U_ctx = rows[1:1 + c]
        U_neg = rows[1 + c:].reshape(c, -1, rows.shape[1])
        l, g_v, g_ctx, g_neg = sgns_loss_grads(v, U_ctx, U_neg, np.ones(c, dtype=bool))
        loss += l
        # one delta row per row occurrence: centre first, then per context its
        # positive output row followed by its negatives
        keys.append([centres[i]])
        deltas.append(-lr * g_v[None, :])
        for j in range(c):
            keys.append([ctx_keys[j]])
            deltas.append(-lr * g_ctx[j][None, :])
            keys.append(neg_keys[j])
            deltas.append(-lr * g_neg[j])
    keys = np.concatenate([np.asarray(k, dtype=np.int64) for k in keys])
    deltas = np.concatenate(deltas)
    pm.push(w, keys, deltas.astype(np.float32))
    return float(loss)
