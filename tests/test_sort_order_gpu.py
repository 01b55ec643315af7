"""The backward's stable radix sort, read back through cb_tbe_sorted_payloads.

Both the GPU sort and the oracle's std::stable_sort order each table's lookups
by row and break ties by lookup position, so the order itself is unique and is
compared bit for bit: with per-sample weights (or mean pooling) the payload is
the lookup position, which must equal the oracle's permutation; without, it is
the lookup's bag, which must equal the bag of the oracle's permutation.
"""

import numpy as np
import pytest
import torch

import oracle
from tests.helpers import bag_of_positions, inject_out_of_range, random_problem, table_meta

pytestmark = pytest.mark.gpu
DEV = torch.device("cuda:0")


def _skewed_problem(seed, weighted, batch=300):
    # Hot rows (many ties), tables of 1 to ~40 radix tiles, rows above 2^16 so
    # that three passes run, and empty bags.
    tables, ind, off, w = random_problem(seed, dims=(16, 64, 128), rows=(3, 5000, 300_000),
                                         batch=batch, max_len=700, weighted=weighted, empty_frac=0.1)
    g = torch.Generator().manual_seed(seed + 1)
    u = torch.rand(ind.numel(), generator=g, dtype=torch.float64)
    rows_of = torch.tensor([t.shape[0] for t in tables])[bag_of_positions(off) // batch]
    ind = torch.floor(rows_of.double() * u ** 6).to(torch.int64)  # heavily skewed toward row 0
    return tables, ind, off, w, batch


def _sorted(tables, batch, ind, off, w, mean, go):
    from paper_2609_30656_gb300.tbe import TBE
    m = TBE([t.to(DEV) for t in tables], pooling="mean" if mean else "sum")
    m.backward(ind.to(DEV), off.to(DEV), go.to(DEV), None if w is None else w.to(DEV))
    got = m.sorted_payloads(ind.numel()).cpu().numpy()
    m.get_error()
    return got


@pytest.mark.parametrize("weighted,mean", [(False, False), (True, False), (False, True)])
def test_sorted_order_is_the_oracles_stable_permutation(weighted, mean):
    tables, ind, off, w, batch = _skewed_problem(61, weighted)
    rows, dims = table_meta(tables)
    go = torch.randn(batch, int(dims.sum()), generator=torch.Generator().manual_seed(62))
    got = _sorted(tables, batch, ind, off, w, mean, go)
    res = oracle.backward(rows, dims, batch, ind, off, go, weights=w, mean=mean)
    # many ties: the order among equal rows is what stability decides
    assert res.num_unique < ind.numel() // 4
    if weighted or mean:
        np.testing.assert_array_equal(got, res.perm)
    else:
        np.testing.assert_array_equal(got, bag_of_positions(off).numpy()[res.perm])


@pytest.mark.parametrize("weighted", [False, True])
def test_out_of_range_lookups_sort_after_their_tables_rows(weighted):
    tables, ind, off, w, batch = _skewed_problem(63, weighted, batch=200)
    bad_ind, bad = inject_out_of_range(tables, ind, off, batch, 64, frac=0.05)
    rows, dims = table_meta(tables)
    go = torch.randn(batch, int(dims.sum()), generator=torch.Generator().manual_seed(65))
    got = _sorted(tables, batch, bad_ind, off, w, False, go)
    # expected: per table, a stable sort on the row with out-of-range lookups
    # given the key rows_t (numpy's stable argsort, not the library's sort)
    bag = bag_of_positions(off).numpy()
    table = bag // batch
    key = np.where(bad.numpy(), rows[table], bad_ind.numpy())
    order = np.lexsort((np.arange(key.size), key, table))
    if weighted:
        np.testing.assert_array_equal(got, order)
    else:
        want = np.where(bad.numpy()[order], 0xFFFFFFFF, bag[order])
        np.testing.assert_array_equal(got, want)


def test_readback_needs_a_backward_of_the_same_size():
    from paper_2609_30656_gb300.tbe import TBE, CbTbeError
    tables, ind, off, w, batch = _skewed_problem(66, False, batch=20)
    m = TBE([t.to(DEV) for t in tables])
    with pytest.raises(CbTbeError):
        m.sorted_payloads(ind.numel())  # no backward yet
    m.forward(ind.to(DEV), off.to(DEV))
    with pytest.raises(CbTbeError):
        m.sorted_payloads(ind.numel())  # a forward sorts nothing
    go = torch.randn(batch, sum(t.shape[1] for t in tables))
    m.backward(ind.to(DEV), off.to(DEV), go.to(DEV))
    with pytest.raises(CbTbeError):
        m.sorted_payloads(ind.numel() + 1)
    assert m.sorted_payloads(ind.numel()).numel() == ind.numel()
