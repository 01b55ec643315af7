"""Seeded input generator: shapes, determinism and distribution statistics (CPU)."""

import math

import numpy as np
import pytest
import torch

from paper_2609_30656_gb300 import workloads as wl


def _sample_lengths(name, count=200_000, seed=0):
    w = wl.get_workload(name)
    return wl.bag_lengths(w, wl._gen("cpu", seed, 99), count, "cpu").numpy().astype(np.float64)


def test_poisson_lengths_mean():
    x = _sample_lengths("cfg2")
    assert x.min() >= 0 and x.max() <= 100
    # Clipping at 100 removes a negligible tail of Poisson(20).
    assert abs(x.mean() - 20.0) < 4 * math.sqrt(20.0 / x.size)


def test_lognormal_lengths_mean_matches_rounded_clipped_analytic():
    w = wl.get_workload("cfg4")
    L = w.lengths
    mu = math.log(L.mean) - 0.5 * L.sigma ** 2

    def cdf(x):
        if x <= 0:
            return 0.0
        return 0.5 * (1 + math.erf((math.log(x) - mu) / (L.sigma * math.sqrt(2))))

    # P(round(X) = k) for k in 1..499; k = 500 absorbs the clipped tail.
    probs = {k: cdf(k + 0.5) - cdf(k - 0.5) for k in range(1, 500)}
    probs[500] = 1 - cdf(499.5)
    mean = sum(k * p for k, p in probs.items())
    var = sum(k * k * p for k, p in probs.items()) - mean ** 2
    x = _sample_lengths("cfg4")
    assert x.min() >= 0 and x.max() <= 500
    assert abs(x.mean() - mean) < 4 * math.sqrt(var / x.size)
    assert 45 < mean < 51


def test_power_law_lengths_mean_and_empty_fraction():
    w = wl.get_workload("cfg5")
    L = w.lengths
    ks = np.arange(L.lo, L.hi + 1, dtype=np.float64)
    p = ks ** -L.alpha
    p /= p.sum()
    mean_nonempty = float((ks * p).sum())
    var_nonempty = float((ks * ks * p).sum()) - mean_nonempty ** 2
    x = _sample_lengths("cfg5", count=400_000)
    empty = (x == 0).mean()
    assert abs(empty - 0.05) < 4 * math.sqrt(0.05 * 0.95 / x.size)
    ne = x[x > 0]
    assert ne.min() >= 7 and ne.max() <= 1000
    assert abs(ne.mean() - mean_nonempty) < 4 * math.sqrt(var_nonempty / ne.size)
    assert 29 < 0.95 * mean_nonempty < 33  # "mean ~30" overall


@pytest.mark.parametrize("N,alpha,k", [(100_000, 1.05, 100), (5_000_000, 1.2, 4900),
                                       (1000, 1.1, 10)])
def test_zipf_head_mass(N, alpha, k):
    ranks = wl.zipf_ranks(N, alpha, 300_000, wl._gen("cpu", 5, N), "cpu").numpy()
    assert ranks.min() >= 0 and ranks.max() < N
    r = np.arange(1, N + 1, dtype=np.float64) ** -alpha
    head = r[:k].sum() / r.sum()
    got = (ranks < k).mean()
    assert abs(got - head) < 4 * math.sqrt(head * (1 - head) / ranks.size)
    # rank 0 is the most frequent
    assert (ranks == 0).mean() == pytest.approx(r[0] / r.sum(), abs=5e-3)


def test_batch_shapes_and_determinism():
    w = wl.scaled(wl.get_workload("cfg2"), num_tables=3, batch=64)
    a = wl.make_batch(w, 0, "cpu")
    b = wl.make_batch(w, 0, "cpu")
    c = wl.make_batch(w, 0, "cpu", batch_index=1)
    assert a.offsets.shape == (3 * 64 + 1,) and a.offsets[0] == 0
    assert int(a.offsets[-1]) == a.indices.numel()
    assert (a.offsets[1:] >= a.offsets[:-1]).all()
    assert torch.equal(a.indices, b.indices) and torch.equal(a.offsets, b.offsets)
    assert not torch.equal(a.offsets, c.offsets)
    for t in range(3):
        s, e = int(a.offsets[t * 64]), int(a.offsets[(t + 1) * 64])
        assert a.indices[s:e].min() >= 0 and a.indices[s:e].max() < w.rows[t]


def test_rank_to_row_map_is_fixed_per_table_and_hot_rows_repeat():
    w = wl.scaled(wl.get_workload("cfg2"), num_tables=2, batch=512)
    a = wl.make_batch(w, 0, "cpu", batch_index=0)
    b = wl.make_batch(w, 0, "cpu", batch_index=1)
    s, e = int(a.offsets[0]), int(a.offsets[512])
    hot_a = torch.bincount(a.indices[s:e], minlength=w.rows[0]).argmax()
    s, e = int(b.offsets[0]), int(b.offsets[512])
    hot_b = torch.bincount(b.indices[s:e], minlength=w.rows[0]).argmax()
    assert hot_a == hot_b  # the same permuted row is hottest in every batch


def test_tables_are_rounded_normal_and_cfg3_rows_are_log_uniform():
    w = wl.scaled(wl.get_workload("cfg4"), num_tables=3, rows=2000)
    tabs = wl.make_tables(w, 0, "cpu")
    assert [t.dtype for t in tabs] == [torch.bfloat16] * 3
    assert [tuple(t.shape) for t in tabs] == [(2000, 64), (2000, 128), (2000, 256)]
    x = torch.cat([t.float().flatten() for t in tabs])
    assert abs(float(x.std()) - 0.01) < 5e-4 and abs(float(x.mean())) < 5e-4
    rows3 = wl.get_workload("cfg3").rows
    assert len(rows3) == 26 and min(rows3) >= 10 and max(rows3) <= 10_000_000
    assert wl.get_workload("cfg3", seed=0).rows == rows3


def test_full_size_shapes_are_as_specified():
    c1, c5 = wl.get_workload("cfg1"), wl.get_workload("cfg5")
    assert (c1.num_tables, c1.rows[0], c1.dims[0], c1.batch) == (1, 1000, 64, 128)
    assert (c5.num_tables, c5.rows[0], c5.dims[0], c5.batch, c5.dtype) == (100, 5_000_000, 128,
                                                                            65536, "f16")
    c4 = wl.get_workload("cfg4")
    assert c4.sum_dims == sum([64, 128, 256][t % 3] for t in range(64)) and c4.weighted and c4.mean
    assert wl.get_workload("cfg5u").zipf_alpha is None


def test_integer_valued_inputs():
    w = wl.scaled(wl.get_workload("cfg4"), num_tables=2, batch=16, rows=100)
    tabs = wl.make_tables(w, 0, "cpu", int_valued=True)
    assert all(float((t.float() - t.float().round()).abs().max()) == 0 for t in tabs)
    bt = wl.make_batch(w, 0, "cpu", int_valued=True)
    assert set(bt.weights.unique().tolist()) <= {0.0, 1.0, 2.0}
    go = wl.make_grad_out(w, 0, "cpu", int_valued=True)
    assert go.abs().max() <= 8
