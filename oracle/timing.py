"""Oracle of adaptive action timing (Sec. 4.2, Algorithm 1).

TEST INFRASTRUCTURE ONLY (see oracle/__init__.py).

The manager acts on intent signals in communication rounds.  It models the
number of clocks worker i advances during one round as Poisson(lambda_i),
estimates lambda_i by exponential smoothing over past rounds, and acts on an
intent in round t when the worker might reach the intent's start before the
next round ends:

    Delta = C_t - C_{t-1}                       (clocks during the last round)
    if Delta > 0:  est_t = (1 - alpha) est_{t-1} + alpha Delta
    else:          est_t = est_{t-1}            (paused workers keep the estimate)
    act  iff  C_start < C_t + Q(2 max(est_t, Delta), p)

Q(lam, p) is the p quantile of Poisson(lam): the smallest integer q with
P(X <= q) >= p.  The paper's settings: alpha = 0.1, p = 0.9999, est_0 = 10.

Arithmetic: fp64.  The quantile adds the probabilities P(X = j) for
j = 0, 1, ... in that order, each computed as exp(-lam + j ln lam - ln j!),
until the sum reaches p (or j passes lam + 64 sqrt(lam) + 64, which no
quantile with p < 1 - 1e-12 reaches: a guard against rounding).
"""
import math

ALPHA = 0.1
P = 0.9999
LAMBDA0 = 10.0


def poisson_quantile(lam, p):
    """Smallest integer q >= 0 with P(X <= q) >= p for X ~ Poisson(lam), lam > 0, 0 < p < 1."""
    if not (lam > 0.0) or not (0.0 < p < 1.0):
        raise ValueError("need lam > 0 and 0 < p < 1")
    ln_lam = math.log(lam)
    qmax = lam + 64.0 * math.sqrt(lam) + 64.0    # far past any quantile with p < 1 - 1e-12
    cdf = 0.0
    q = 0
    while True:
        cdf += math.exp(-lam + q * ln_lam - math.lgamma(q + 1.0))
        if cdf >= p or q >= qmax:
            return q
        q += 1


class RateEstimate:
    """Per-worker state of Algorithm 1: the estimate and the clock at the start of the previous round."""

    def __init__(self, lambda0=LAMBDA0, alpha=ALPHA, p=P):
        self.est = float(lambda0)
        self.prev_clock = 0
        self.alpha = float(alpha)
        self.p = float(p)

    def round(self, clock):
        """Start of a round at worker clock `clock`: update the estimate and return the action bound b.

        In this round the manager acts on every intent with C_start < clock + b."""
        delta = clock - self.prev_clock
        if delta > 0:
            self.est = (1.0 - self.alpha) * self.est + self.alpha * delta
        self.prev_clock = clock
        return poisson_quantile(2.0 * max(self.est, float(delta)), self.p)
