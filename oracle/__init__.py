"""Plain, slow CPU oracle of AdaPM's intent-driven parameter access.

TEST INFRASTRUCTURE ONLY.  Nothing in the product path imports, calls or
executes this package: only tests/, __graft_entry__.smoke() and the
cpu_baseline / reference legs of bench.py use it.  It shares no code with
the CUDA library (paper_2206_00470_gb300/); both are fed from the seeded
input generators in synth/, which hold none of the method's arithmetic.

Modules
  store  intent windows, replica lifetime, pull, push, sync (Sec. 3, Sec. 4.1,
         App. B.1.2, Sec. 5.1 consistency model); optionally the relocation
         rule of Sec. 4.1 / App. B.2.4
  timing adaptive action timing (Sec. 4.2, Algorithm 1): the Poisson quantile
         and the per-worker rate estimate
  steps  the three training steps (App. C: MF, ComplEx KGE, skip-gram WV)
  driver the per-clock loop of a data-parallel worker (Fig. 2 pattern)

Precision: the parameter store holds fp32 values (the workloads fix fp32
parameters); every arithmetic step (sums of deltas, merges, losses and
gradients) is carried out in fp64 and rounded to fp32 once, when stored.

Pins (tests/test_oracle_*.py): brute-force active sets from the raw call log,
the sum invariant with dyadic deltas (bit-exact), hand-worked scenarios in
tests/golden/, the owner and replica intervals of the paper's Fig. 4b-d and
Fig. 10a, the owner recomputed by brute force from the call log, the
Poisson quantile against scipy's, the rate estimate against the closed form
of its recursion, the versioned refresh equal to the full one in exact
arithmetic, the
single-worker reduction to textbook mini-batch SGD and to textbook mini-batch
AdaGrad, one AdaGrad step per occurrence of a repeated key (hand numbers and
per-occurrence finite differences),
fp64 finite-difference gradients, ComplEx scores by complex arithmetic and
closed forms, Zipf frequencies by chi-square.  No function here is "parity
unpinned".
"""
from .store import ParameterManagerOracle, OracleError  # noqa: F401
