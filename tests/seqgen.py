"""Seeded random call sequences for differential tests (inputs only).

A sequence is a list of dicts {"op": ..., ...} over the public calls
intent / advance / pull / push / sync.  Intents include overlapping,
late (start < clock), empty (end <= start) and already-expired windows and
repeated keys; pushes include repeated keys and keys without a replica.
Deltas are dyadic (multiples of 2^-10, |d| <= 1/16) unless gaussian=True,
so that sums are exact in fp32 whatever their order.
"""
import numpy as np


def random_sequence(seed, num_keys, value_len, num_workers, n_ops, max_batch=12,
                    gaussian=False, max_ahead=3, max_span=4, key_pool=None):
    rng = np.random.default_rng(seed)
    clocks = [0] * num_workers
    pool = np.arange(num_keys) if key_pool is None else np.asarray(key_pool)
    ops = []
    for _ in range(n_ops):
        r = rng.random()
        w = int(rng.integers(num_workers))
        if r < 0.3:
            n = int(rng.integers(0, max_batch + 1))
            keys = rng.choice(pool, size=n, replace=True)
            kind = rng.random()
            c = clocks[w]
            if kind < 0.6:
                s = c + int(rng.integers(0, max_ahead + 1))
                e = s + int(rng.integers(1, max_span + 1))
            elif kind < 0.75:      # late: started in the past, still open
                s = c - int(rng.integers(1, 3))
                e = c + int(rng.integers(1, 3))
            elif kind < 0.9:       # empty window
                s = c + int(rng.integers(0, 3))
                e = s - int(rng.integers(0, 2))
            else:                  # already expired
                e = c - int(rng.integers(0, 2))
                s = e - int(rng.integers(1, 3))
            ops.append({"op": "intent", "w": w, "keys": keys, "start": s, "end": e})
        elif r < 0.5:
            ops.append({"op": "advance", "w": w})
            clocks[w] += 1
        elif r < 0.7:
            n = int(rng.integers(0, max_batch + 1))
            ops.append({"op": "pull", "w": w, "keys": rng.choice(pool, size=n, replace=True)})
        elif r < 0.92:
            n = int(rng.integers(0, max_batch + 1))
            keys = rng.choice(pool, size=n, replace=True)
            if gaussian:
                d = rng.normal(0.0, 1e-3, size=(n, value_len)).astype(np.float32)
            else:
                d = (rng.integers(-64, 65, size=(n, value_len)) * 2.0 ** -10).astype(np.float32)
            ops.append({"op": "push", "w": w, "keys": keys, "deltas": d})
        else:
            ops.append({"op": "sync"})
    return ops


def dyadic_init(num_keys, value_len, seed):
    rng = np.random.default_rng(seed + 991)
    return (rng.integers(-1024, 1025, size=(num_keys, value_len)) * 2.0 ** -10).astype(np.float32)
