"""Oracle of a data-parallel worker loop driven by intent signals (Fig. 2).

TEST INFRASTRUCTURE ONLY (see oracle/__init__.py).

The data loader of worker w signals Intent(P_j, j, j + span) for batch j as
soon as the batch is built, `lookahead` clocks before the worker trains on
it (Fig. 2: after batch i is constructed the loader signals intent for the
parameters P_i of batch i).  One clock of the whole job:

    for w = 0 .. W-1:
        Intent(P_{c+L}, c+L, c+L+span)     (loader runs L batches ahead)
        work(w, c)                          (pull + step + push of batch c)
        advanceClock()
    sync()

At the start every worker signals the first L batches.  Workers are run in
ascending order; every key a worker touches in its own step has a replica at
that worker, so the order does not change any value.
"""


def start(pm, workers, lookahead, span, keys_of):
    for w in range(workers):
        for j in range(lookahead):
            pm.intent(w, keys_of(w, j), j, j + span)


def clock(pm, workers, lookahead, span, c, keys_of, work):
    """One clock; returns [work(w, c) for each worker]."""
    out = []
    for w in range(workers):
        j = c + lookahead
        pm.intent(w, keys_of(w, j), j, j + span)
        out.append(work(w, c))
        pm.advance_clock(w)
    pm.sync()
    return out
