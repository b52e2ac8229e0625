"""Input generators: exact Zipf frequencies, bijective key maps, reproducible init rows."""
import math

import numpy as np
import pytest
import torch

from synth import hashgen, workloads as wl
from synth.zipf import affine_perm_params, ranks_to_keys, zipf_pmf, zipf_ranks


@pytest.mark.parametrize("s", [0.0, 0.75, 1.0, 1.1, 1.4])
def test_zipf_frequencies_chi_square(s):
    N, n = 40, 200_000
    r = zipf_ranks(n, N, s, torch.Generator().manual_seed(3))
    counts = np.bincount(r.numpy(), minlength=N)
    p = np.array(zipf_pmf(N, s))
    chi2 = float(((counts - n * p) ** 2 / (n * p)).sum())
    # 39 degrees of freedom: P(chi2 > 80) < 1e-4
    assert chi2 < 80.0, chi2
    assert r.min() >= 0 and r.max() < N


def test_zipf_large_n_head_probability():
    # P(rank 0) = 1 / H_{N,s}; checks the sampler on a 10^8 range
    N, s, n = 10 ** 8, 1.1, 400_000
    r = zipf_ranks(n, N, s, torch.Generator().manual_seed(4))
    h = sum(k ** -s for k in range(1, 200_001)) + ((N + 0.5) ** (1 - s) - (200_000.5) ** (1 - s)) / (1 - s)
    p0 = 1.0 / h
    got = float((r == 0).double().mean())
    assert abs(got - p0) < 5 * math.sqrt(p0 * (1 - p0) / n)
    assert int(r.max()) < N


def test_rank_to_key_is_a_bijection():
    for N in (1, 7, 1000, 1500, 700_000):
        a, _ = affine_perm_params(N, 0)
        assert math.gcd(a, N) == 1
        if N <= 700_000:
            k = ranks_to_keys(torch.arange(N), N, 5)
            assert torch.unique(k).numel() == N and int(k.min()) == 0 and int(k.max()) == N - 1


def test_init_rows_identical_on_numpy_and_torch_paths():
    keys = np.array([0, 1, 5, 123_456, 99_999_999], dtype=np.int64)
    a = hashgen.init_rows_np(keys, 12, 8, seed=3, std=0.1)
    t = torch.tensor(keys).view(-1, 1)
    cols = torch.arange(8).view(1, -1)
    b = hashgen.normal_ih4_torch(t, cols, 3, 0.1).numpy()
    assert np.array_equal(a[:, :8], b) and not a[:, 8:].any()
    whole = hashgen.init_store_torch(64, 12, 8, 3, 0.1, "cpu", chunk_rows=10)
    assert np.array_equal(whole.numpy(), hashgen.init_rows_np(np.arange(64), 12, 8, 3, 0.1))
    d = hashgen.init_rows_np(keys, 4, 4, 1, 0.0, kind="dyadic")
    assert np.array_equal(d * 1024, np.round(d * 1024)) and np.abs(d).max() <= 1.0


def test_init_rows_moments():
    x = hashgen.init_store_torch(1 << 15, 16, 16, 0, 0.1, "cpu")
    assert abs(float(x.mean())) < 1e-3 and abs(float(x.std()) - 0.1) < 1e-3


def test_workload_batches_are_reproducible_and_in_range():
    mf = wl.MF
    r1, c1, v1 = wl.mf_batch(mf, 3, 7, batch=512)
    r2, c2, v2 = wl.mf_batch(mf, 3, 7, batch=512)
    assert torch.equal(r1, r2) and torch.equal(c1, c2) and torch.equal(v1, v2)
    assert (r1 % mf.workers == 3).all() and int(r1.max()) < mf.rows
    assert int(c1.min()) >= mf.rows and int(c1.max()) < mf.num_keys
    h, r, t, n = wl.complex_batch(wl.COMPLEX, 0, 0, batch=64)
    assert int(r.min()) >= wl.COMPLEX.entities and int(r.max()) < wl.COMPLEX.num_keys
    assert n.shape == (64, 100) and int(n.max()) < wl.COMPLEX.entities
    k = wl.micro_keys(wl.MICRO, 2, 9, batch=4096)
    assert int(k.max()) < wl.MICRO.num_keys and torch.equal(k, wl.micro_keys(wl.MICRO, 2, 9, batch=4096))


def test_sgns_batch_windows():
    import dataclasses
    cfg = dataclasses.replace(wl.SGNS, batch=64, total_tokens=64 * 8 * 4)
    cen, ctx, neg = wl.sgns_batch(cfg, 1, 0)
    assert ctx.shape == (64, 10) and neg.shape == (64, 10, 25)
    # first centre of the shard has no left context
    assert (ctx[0, :5] == wl.MISSING).all() and (ctx[0, 5:] != wl.MISSING).all()
    # interior: context at offset +1 is the next centre
    assert torch.equal(ctx[:-1, 5], cen[1:])
    cen3, ctx3, _ = wl.sgns_batch(cfg, 1, 3)             # last chunk of the shard
    assert (ctx3[-1, 5:] == wl.MISSING).all()
