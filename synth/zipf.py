"""Exact Zipf(s) sampling over ranks 1..N and a seeded rank -> key permutation.

Sampler: rejection-inversion for monotone discrete distributions
(W. Hoermann and G. Derflinger, "Rejection-inversion to generate variates
from monotone discrete distributions", ACM TOMACS 6(3), 1996), specialised
to P(k) proportional to k^-s, k = 1..N.  With the hat h(x) = x^-s and its
antiderivative H, a uniform u on (H(1.5) - 1, H(N + 0.5)] is inverted to
x = H^-1(u) and rounded to k; k is accepted when u lies in the top h(k) of
k's interval [H(k - 0.5), H(k + 0.5)], which makes every k appear with
probability proportional to h(k) exactly.  A squeeze (k - x <= 2 -
H^-1(H(2.5) - h(2))) accepts most draws without evaluating H.  s = 0 is the
uniform distribution.  Works for any s >= 0, any N >= 1, in float64, on torch
CPU and CUDA tensors alike (the two backends draw different uniforms, so use
one backend for data that must match).

Rank -> key: key = (a * (rank - 1) + b) mod N with gcd(a, N) = 1, a and b
derived from a seed: a bijection of [0, N) that keeps hot ranks apart.
"""
import math

import torch


def _expm1_over(t):
    # (exp(t) - 1) / t, continuous at t = 0
    small = t.abs() < 1e-8
    safe = torch.where(small, torch.ones_like(t), t)
    return torch.where(small, 1.0 + 0.5 * t, torch.expm1(safe) / safe)


def _log1p_over(t):
    # log(1 + t) / t, continuous at t = 0
    small = t.abs() < 1e-8
    safe = torch.where(small, torch.ones_like(t), t)
    return torch.where(small, 1.0 - 0.5 * t, torch.log1p(safe) / safe)


class _ZipfHat:
    def __init__(self, n, s):
        self.n = int(n)
        self.s = float(s)

    def h(self, x):
        return torch.exp(-self.s * torch.log(x))

    def H(self, x):
        lx = torch.log(x)
        return _expm1_over((1.0 - self.s) * lx) * lx

    def H_inv(self, y):
        t = torch.clamp(y * (1.0 - self.s), min=-1.0)
        return torch.exp(_log1p_over(t) * y)


def zipf_ranks(n, N, s, generator, device="cpu"):
    """n samples of a Zipf(s) rank in [0, N) (rank 0 is the most frequent)."""
    n = int(n)
    if n == 0:
        return torch.empty(0, dtype=torch.int64, device=device)
    if s == 0.0 or N == 1:
        return torch.randint(0, N, (n,), generator=generator, device=device, dtype=torch.int64)
    hat = _ZipfHat(N, s)
    f64 = dict(dtype=torch.float64, device=device)
    one = torch.ones((), **f64)
    h_x1 = float(hat.H(1.5 * one) - 1.0)
    h_n = float(hat.H((N + 0.5) * one))
    squeeze = float(2.0 - hat.H_inv(hat.H(2.5 * one) - hat.h(2.0 * one)))
    out = torch.empty(n, dtype=torch.int64, device=device)
    todo = torch.arange(n, device=device)
    while todo.numel() > 0:
        m = todo.numel()
        u = torch.rand(m, generator=generator, **f64)
        u = h_n + u * (h_x1 - h_n)
        x = hat.H_inv(u)
        k = torch.clamp(torch.floor(x + 0.5), 1.0, float(N))
        accept = (k - x <= squeeze) | (u >= hat.H(k + 0.5) - hat.h(k))
        out[todo[accept]] = k[accept].to(torch.int64) - 1
        todo = todo[~accept]
    return out


def zipf_pmf(N, s):
    """Exact probabilities of ranks 0..N-1 (float64 list) for tests."""
    w = [(k + 1) ** (-float(s)) for k in range(N)]
    z = math.fsum(w)
    return [x / z for x in w]


def affine_perm_params(N, seed):
    """(a, b) with gcd(a, N) = 1 for the bijection r -> (a r + b) mod N."""
    N = int(N)
    if N <= 1:
        return 1, 0
    g = torch.Generator().manual_seed(int(seed) * 7919 + 17)
    a = int(torch.randint(N // 3 + 1, max(N // 3 + 2, (2 * N) // 3 + 1), (1,), generator=g)) | 1
    while math.gcd(a, N) != 1:
        a += 2
    b = int(torch.randint(0, N, (1,), generator=g))
    return a % N if a % N else 1, b


def ranks_to_keys(ranks, N, seed):
    """Apply the seeded bijection of [0, N) to rank tensors (int64)."""
    a, b = affine_perm_params(N, seed)
    return (ranks * a + b) % N
