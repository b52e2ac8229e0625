"""Seeded synthetic inputs shared by the oracle's tests, the GPU tests and the bench.

This package generates inputs only: keys, data points, delta rows and the
initial parameter store.  It holds none of the parameter manager's arithmetic
(no intent windows, replica rules, sums or gradients), so the oracle and the
CUDA path can both be fed from it without sharing any method code.

Modules
  hashgen    counter-based integer hash -> exactly reproducible init values on
             CPU (numpy) and GPU (torch) alike
  zipf       exact Zipf(s) sampling by rejection-inversion, rank->key permutation
  workloads  the five workload configurations and their per-clock batches
"""
