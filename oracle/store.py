"""Oracle of the parameter manager: intents, replicas, pull, push, sync.

TEST INFRASTRUCTURE ONLY (see oracle/__init__.py).

State follows the paper's description of AdaPM with worker slots in the role
of nodes.  By default replication is always chosen (the paper's "AdaPM w/o
relocation" variant, Sec. 5.5); with relocation=True the full decision rule
of Sec. 4.1 applies (see "Relocation" below):

  main[K][D]        the main copy of every parameter (fp32)
  clock[w]          worker w's logical clock C^w, starts at 0 (Sec. 3)
  intents[w]        recorded Intent(keys, C_start, C_end) calls of worker w
  replicas[w][k]    (val[D], acc[D]) for every key with a replica at w;
                    val is the worker's local copy, acc the updates it wrote
                    since the replica was created or last refreshed

Definitions
  * An intent is active while C_start <= C^w < C_end, inactive before,
    expired after (Sec. 3).  A key is in the active set A_w(c) when some
    recorded intent of w containing it is active at c.  Keys inside one call
    are a set: repeats count once.
  * Replica lifetime (Sec. 4.1): a replica exists for exactly the span in
    which the worker has active intent.  After every call R_w = A_w(C^w).
    Replicas are destroyed before new ones are created, each in ascending
    key order; a key that stays active keeps its replica untouched, which is
    how one intent extends another (Sec. 3).
  * Creating a replica copies main[k] and zeroes acc; destroying one merges
    acc into main[k] (App. B.1.2: replica holders send their updates to the
    owner).
  * pull: a key with a replica at w reads the local copy; any other key reads
    the main copy, which is always current (Sec. 5.1; intent is optional,
    Sec. 4).
  * push: the rows of each distinct key are summed in order of appearance and
    added to both val and acc of w's replica, or to main when w holds none.
  * sync: for every key with at least one replica, main[k] += sum over the
    holders (ascending worker) of acc, then every holder's val = main[k] and
    acc = 0 (App. B.1.2: the owner merges the updates and propagates them to
    the replica holders; sending only unseen versions gives the same values).

Versioned refresh (App. B.1.2: holders request only the updates they have
not received).  With delta_refresh=True, sync leaves the value of a replica
alone when its holder is the key's only holder and nobody else wrote main[k]
since the last sync that merged k or the last replica creation of k (no
write to main without a replica, no destroyed replica): the holder has all
the updates already, its own.  Its
pending updates are still merged and cleared.  In exact arithmetic nothing
changes; in fp32 the holder keeps its own rounding of the same sum.

Action timing (Sec. 4.2).  action_timing="start" (default) acts on an intent
exactly when it becomes active.  "signal" acts when the intent is signalled
(the paper's immediate-action ablation, Sec. 5.8): its window is treated as
starting at the signalling clock.  "adaptive" follows Algorithm 1
(oracle/timing.py): every sync is a communication round; after its merge,
each worker's intents that Algorithm 1 selects are treated as active from
that round on; an intent no round selected becomes active at its start.

Relocation (Sec. 4.1 and App. B.2.4, "relocate only when exactly one node has
active intent"; scenarios of Fig. 4b-d and Fig. 10a)
  * Every key has an owner: a worker slot, or its home (-1) before any
    worker has held it.  The owner accesses the main copy directly and holds
    no replica; every other worker with active intent holds a replica.
  * Whenever exactly one worker has active intent for a key and it is not the
    owner, the key is relocated to it: if that worker holds a replica, the
    replica is destroyed first (its pending updates merged into main, as on
    any destruction), then the worker becomes the owner.  Ownership stays
    where it is when the owner's intent expires, while several workers have
    active intent, and while nobody has.
  * Within one call only the calling worker's active set changes, so a key
    is either joined or left by that worker.  Left keys (ascending) go first:
    the worker's replica is destroyed, then a sole remaining active worker
    becomes the owner.  Joined keys (ascending) follow: with no other active
    worker the caller becomes the owner, otherwise it gets a replica unless
    it is the owner already.
  * pull, push and sync are unchanged: the owner holds no replica, so its
    reads and writes go to main; a sole active worker therefore sees other
    workers' writes at once.

Arithmetic: every sum runs in fp64 and is rounded to fp32 once when stored.
"""
import numpy as np

from .timing import RateEstimate


class OracleError(ValueError):
    """An argument the parameter manager must reject (bad worker, key out of range)."""


def _f32(x):
    return np.asarray(x, dtype=np.float64).astype(np.float32)


class ParameterManagerOracle:
    def __init__(self, num_keys, value_len, num_workers, init, relocation=False, action_timing="start",
                 timing_alpha=None, timing_p=None, timing_lambda0=None, delta_refresh=False):
        init = np.asarray(init, dtype=np.float32)
        if init.shape != (num_keys, value_len):
            raise OracleError("init must have shape (num_keys, value_len)")
        self.K = int(num_keys)
        self.D = int(value_len)
        self.W = int(num_workers)
        self.relocation = bool(relocation)
        self.main = init.copy()
        self.clock = [0] * self.W
        self.intents = [[] for _ in range(self.W)]   # entries: (frozenset keys, start, end)
        self.replicas = [dict() for _ in range(self.W)]
        self.active = [set() for _ in range(self.W)]  # A_w(C^w) as of w's last call
        self.owner = np.full(self.K, -1, dtype=np.int64)
        self.created = self.destroyed = self.relocations = 0
        if action_timing not in ("start", "adaptive", "signal"):
            raise OracleError("action_timing must be 'start', 'adaptive' or 'signal'")
        self.action_timing = action_timing
        kw = {k: v for k, v in (("alpha", timing_alpha), ("p", timing_p), ("lambda0", timing_lambda0))
              if v is not None}
        self.rates = [RateEstimate(**kw) for _ in range(self.W)]
        self.delta_refresh = bool(delta_refresh)
        self.changed = np.zeros(self.K, dtype=bool)   # main[k] written other than by a sync merge
        self.refreshed = 0

    # -- argument checks ---------------------------------------------------
    def _check_worker(self, w):
        if not (0 <= w < self.W):
            raise OracleError(f"worker {w} out of range")

    def _check_keys(self, keys):
        keys = np.asarray(keys, dtype=np.int64).reshape(-1)
        if keys.size and (keys.min() < 0 or keys.max() >= self.K):
            raise OracleError("key out of range")
        return keys

    # -- intent windows (Sec. 3) --------------------------------------------
    def _is_active(self, start, end, c):
        return start <= c < end

    def active_set(self, w, c=None):
        c = self.clock[w] if c is None else c
        out = set()
        for keys, s, e in self.intents[w]:
            if self._is_active(s, e, c):
                out |= keys
        return out

    def refcount(self, w, k):
        """Number of w's intent calls that are active now and contain k."""
        c = self.clock[w]
        return sum(1 for keys, s, e in self.intents[w] if self._is_active(s, e, c) and k in keys)

    def _create(self, w, k):
        self.replicas[w][k] = (self.main[k].copy(), np.zeros(self.D, dtype=np.float32))
        # a new replica has seen every update; a replica of another worker that has not is refreshed at
        # the next sync anyway, since the key then has several holders, or becomes the only one by the
        # destruction of this one, which marks the key again
        self.changed[k] = False
        self.created += 1

    def _destroy(self, w, k):
        val, acc = self.replicas[w].pop(k)
        self.main[k] = _f32(self.main[k].astype(np.float64) + acc.astype(np.float64))
        self.changed[k] = True
        self.destroyed += 1

    def _relocate(self, k, w):
        """Make w the owner of k; a replica it holds is merged into main first."""
        if self.owner[k] == w:
            return
        if k in self.replicas[w]:
            self._destroy(w, k)
        self.owner[k] = w
        self.relocations += 1

    def _others_active(self, w, k):
        return [v for v in range(self.W) if v != w and k in self.active[v]]

    def _reconcile(self, w):
        now = self.active_set(w)
        if self.relocation:
            before = self.active[w]
            for k in sorted(before - now):            # w's intent for k expired
                if k in self.replicas[w]:
                    self._destroy(w, k)
                others = self._others_active(w, k)
                if len(others) == 1:
                    self._relocate(k, others[0])
            for k in sorted(now - before):            # w's intent for k became active
                others = self._others_active(w, k)
                if not others:
                    self._relocate(k, w)
                elif self.owner[k] != w:
                    self._create(w, k)
        else:
            # R_w := A_w(C^w): destroy, then create, each in ascending key order
            held = set(self.replicas[w])
            for k in sorted(held - now):
                self._destroy(w, k)
            for k in sorted(now - held):
                self._create(w, k)
        self.active[w] = now
        # expired intents can never become active again (clocks only rise)
        c = self.clock[w]
        self.intents[w] = [(keys, s, e) for keys, s, e in self.intents[w] if e > c]

    def intent(self, w, keys, start, end):
        """Intent(keys, C_start, C_end) of worker w; the optional type is not modelled."""
        self._check_worker(w)
        keys = self._check_keys(keys)
        start, end = int(start), int(end)
        if end <= start or end <= self.clock[w]:
            return                      # empty or already expired window: nothing to do
        if self.action_timing == "signal":
            start = min(start, self.clock[w])   # act as soon as the intent is signalled
        self.intents[w].append((frozenset(int(k) for k in keys), start, end))
        self._reconcile(w)              # activates now if start <= C^w

    def advance_clock(self, w):
        self._check_worker(w)
        self.clock[w] += 1
        self._reconcile(w)

    # -- access ----------------------------------------------------------------
    def pull(self, w, keys):
        self._check_worker(w)
        keys = self._check_keys(keys)
        out = np.empty((keys.size, self.D), dtype=np.float32)
        reps = self.replicas[w]
        for i, k in enumerate(keys.tolist()):
            out[i] = reps[k][0] if k in reps else self.main[k]
        return out

    def push(self, w, keys, deltas):
        self._check_worker(w)
        keys = self._check_keys(keys)
        deltas = np.asarray(deltas, dtype=np.float32).reshape(keys.size, self.D)
        groups = {}
        for i, k in enumerate(keys.tolist()):
            groups.setdefault(k, []).append(i)
        reps = self.replicas[w]
        for k in sorted(groups):
            s = np.zeros(self.D, dtype=np.float64)
            for i in groups[k]:                      # order of appearance
                s += deltas[i].astype(np.float64)
            if k in reps:
                val, acc = reps[k]
                reps[k] = (_f32(val.astype(np.float64) + s), _f32(acc.astype(np.float64) + s))
            else:
                self.main[k] = _f32(self.main[k].astype(np.float64) + s)
                self.changed[k] = True

    def sync(self):
        keys = sorted(set().union(*[set(r) for r in self.replicas]))
        for k in keys:
            total = self.main[k].astype(np.float64)
            holders = [w for w in range(self.W) if k in self.replicas[w]]
            for w in holders:                        # ascending worker
                total = total + self.replicas[w][k][1].astype(np.float64)
            self.main[k] = _f32(total)
            # versioned refresh: a sole holder of a key nobody else wrote since the last sync has
            # received every update already (its own), so only its pending updates are cleared
            stale = not self.delta_refresh or len(holders) > 1 or self.changed[k]
            for w in holders:
                val = self.main[k].copy() if stale else self.replicas[w][k][0]
                self.replicas[w][k] = (val, np.zeros(self.D, dtype=np.float32))
            self.refreshed += len(holders) if stale else 0
            self.changed[k] = False
        if self.action_timing == "adaptive":
            self._act_in_round()

    def _act_in_round(self):
        """A communication round (one sync) acts on the intents Algorithm 1 selects, worker by worker.

        After the merge (App. B.2.2: the owner merges the updates, then answers the intent signals), every
        recorded intent of worker w that is not active yet and starts before C^w + b_w is treated as active
        from now on; intents no round selected still become active at their start clock."""
        for w in range(self.W):
            c = self.clock[w]
            bound = self.rates[w].round(c)
            acted = False
            for i, (keys, s, e) in enumerate(self.intents[w]):
                if c < s < c + bound:
                    self.intents[w][i] = (keys, c, e)
                    acted = True
            if acted:
                self._reconcile(w)

    # -- inspection --------------------------------------------------------------
    def replica_keys(self, w):
        self._check_worker(w)
        return np.array(sorted(self.replicas[w]), dtype=np.int64)

    def replica_values(self, w):
        """(keys ascending, val rows, acc rows) of worker w's replicas."""
        ks = self.replica_keys(w)
        val = np.array([self.replicas[w][k][0] for k in ks.tolist()], dtype=np.float32).reshape(-1, self.D)
        acc = np.array([self.replicas[w][k][1] for k in ks.tolist()], dtype=np.float32).reshape(-1, self.D)
        return ks, val, acc

    def refcounts(self, w, keys):
        self._check_worker(w)
        keys = self._check_keys(keys)
        return np.array([self.refcount(w, int(k)) for k in keys], dtype=np.int64)

    def read_main(self, keys):
        keys = self._check_keys(keys)
        return self.main[keys].copy()

    def owners(self, keys):
        """Owner worker of each key, -1 for a key still at its home."""
        keys = self._check_keys(keys)
        return self.owner[keys].copy()
