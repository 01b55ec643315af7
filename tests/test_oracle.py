"""Pins for the fp64 CPU oracle (CPU only).

Each pin ties the oracle to something other than itself: hand-worked values
(tests/golden), the IEEE 754 / bfloat16 format definitions as implemented by
numpy and torch, torch's float64 embedding_bag and autograd, brute-force
enumeration, closed-form invariants and the adjoint identity. A dropped term,
a wrong sign, a transposed index or a misplaced column block fails at least
one of them.
"""

import itertools

import numpy as np
import pytest
import torch

import oracle
from tests.conftest import parse_value
from tests.helpers import (random_problem, sparse_to_dense, table_meta, torch_dense_grad_f64,
                           torch_forward_f64)


# ---------------------------------------------------------------- format decoders

def test_half_decoder_matches_ieee_binary16_on_every_bit_pattern():
    bits = np.arange(65536, dtype=np.uint32).astype(np.uint16)
    want = bits.view(np.float16).astype(np.float64)
    got = np.array([oracle.half_to_double(int(b)) for b in bits])
    same = (got == want) | (np.isnan(got) & np.isnan(want))
    assert same.all()
    # signed zeros keep their sign
    assert np.signbit(oracle.half_to_double(0x8000))


def test_bf16_decoder_matches_torch_on_every_bit_pattern():
    bits = torch.arange(65536, dtype=torch.int32).to(torch.int16)
    want = bits.view(torch.bfloat16).to(torch.float64).numpy()
    got = np.array([oracle.bf16_to_double(b) for b in range(65536)])
    same = (got == want) | (np.isnan(got) & np.isnan(want))
    assert same.all()


# ---------------------------------------------------------------- hand-worked values

def _golden_problem(golden):
    g = golden("two_tables_hand.json")
    tables = [np.array(t, dtype=np.float32) for t in g["tables"]]
    ind = np.array(g["indices"], dtype=np.int64)
    off = np.array(g["offsets"], dtype=np.int64)
    w = np.array(g["weights"], dtype=np.float32)
    go = np.array(g["grad_out"], dtype=np.float32)
    return g, tables, ind, off, w, go


@pytest.mark.parametrize("case", ["sum", "mean", "weighted_sum", "weighted_mean"])
def test_forward_hand_worked(golden, case):
    g, tables, ind, off, w, _ = _golden_problem(golden)
    want = np.array([[parse_value(v) for v in row] for row in g["forward"][case]])
    got = oracle.forward(tables, g["batch"], ind, off,
                         weights=w if case.startswith("weighted") else None,
                         mean=case.endswith("mean"))
    np.testing.assert_allclose(got, want, rtol=1e-15, atol=0)


@pytest.mark.parametrize("case", ["sum", "weighted_mean"])
def test_backward_hand_worked(golden, case):
    g, tables, ind, off, w, go = _golden_problem(golden)
    rows, dims = table_meta([torch.from_numpy(t) for t in tables])
    res = oracle.backward(rows, dims, g["batch"], ind, off, go,
                          weights=w if case == "weighted_mean" else None,
                          mean=case == "weighted_mean")
    b = g["backward"]
    assert res.uniq.tolist() == b["uniq"]
    assert res.seg_start.tolist() == b["seg_start"]
    assert res.perm.tolist() == b["perm"]
    assert res.table_offsets.tolist() == b["table_offsets"]
    assert res.grad_offsets.tolist() == b["grad_offsets"]
    np.testing.assert_allclose(res.grads, np.array(b[case], dtype=np.float64), rtol=1e-15,
                               atol=1e-15)


def test_half_storage_hand_worked(golden):
    g = golden("half_storage_hand.json")
    t16 = np.array(g["fp16_rows_bits"], dtype=np.uint16).view(np.float16)
    bag = g["fp16_bag"]
    got = oracle.forward([t16], 1, np.array(bag, np.int64), np.array([0, len(bag)], np.int64))
    np.testing.assert_array_equal(got[0], [parse_value(v) for v in g["fp16_sum"]])

    tb = torch.tensor(g["bf16_rows_bits"], dtype=torch.int32).to(torch.int16).view(torch.bfloat16)
    bag = g["bf16_bag"]
    got = oracle.forward([tb], 1, np.array(bag, np.int64), np.array([0, len(bag)], np.int64),
                         mean=True)
    np.testing.assert_allclose(got[0], [parse_value(v) for v in g["bf16_mean"]], rtol=1e-15,
                               atol=0)


# ---------------------------------------------------------------- library special case

@pytest.mark.parametrize("dtype", [torch.float32, torch.float16, torch.bfloat16])
@pytest.mark.parametrize("weighted,mean", [(False, False), (False, True), (True, False),
                                           (True, True)])
def test_forward_integer_tables_equal_torch_embedding_bag_exactly(dtype, weighted, mean):
    # Integer tables and weights make every partial sum exact, so any correct
    # summation order gives the same bits; mean divides the same exact sum.
    tables, ind, off, w = random_problem(11, dtype=dtype, int_valued=True, weighted=weighted)
    want = torch_forward_f64(tables, 9, ind, off, w, mean).numpy()
    got = oracle.forward(tables, 9, ind, off, weights=w, mean=mean)
    np.testing.assert_array_equal(got, want)


@pytest.mark.parametrize("weighted,mean", [(False, False), (True, True), (False, True)])
def test_forward_random_tables_match_torch_f64(weighted, mean):
    tables, ind, off, w = random_problem(5, weighted=weighted, max_len=40)
    want = torch_forward_f64(tables, 9, ind, off, w, mean).numpy()
    got = oracle.forward(tables, 9, ind, off, weights=w, mean=mean)
    np.testing.assert_allclose(got, want, rtol=1e-12, atol=1e-14)


@pytest.mark.parametrize("weighted,mean", [(False, False), (True, False), (True, True),
                                           (False, True)])
def test_backward_matches_torch_autograd_and_direct_scatter(weighted, mean):
    tables, ind, off, w = random_problem(7, weighted=weighted, max_len=30)
    rows, dims = table_meta(tables)
    go = torch.randn(9, int(dims.sum()), generator=torch.Generator().manual_seed(3))
    res = oracle.backward(rows, dims, 9, ind, off, go, weights=w, mean=mean)
    from_sparse = sparse_to_dense(res, rows, dims)
    direct = oracle.backward_dense(rows, dims, 9, ind, off, go, weights=w, mean=mean)
    auto = torch_dense_grad_f64(tables, 9, ind, off, go, w, mean)
    for a, b, c in zip(from_sparse, direct, auto):
        np.testing.assert_array_equal(a, b)  # same terms, same order
        np.testing.assert_allclose(a, c.numpy(), rtol=1e-12, atol=1e-13)


# ---------------------------------------------------------------- brute force

def test_forward_brute_force_enumeration_of_all_tiny_bags():
    # Every bag of length <= 2 over a 3-row, dim-4 table, written one bag per
    # batch slot, against a direct sum computed here row by row.
    E = np.arange(12, dtype=np.float32).reshape(3, 4) - 5.5
    bags = [()] + [(r,) for r in range(3)] + list(itertools.product(range(3), repeat=2))
    ind = np.array([r for bag in bags for r in bag], dtype=np.int64)
    off = np.concatenate([[0], np.cumsum([len(b) for b in bags])]).astype(np.int64)
    got = oracle.forward([E], len(bags), ind, off)
    for b, bag in enumerate(bags):
        want = np.zeros(4)
        for r in bag:
            want += E[r].astype(np.float64)
        np.testing.assert_array_equal(got[b], want)


# ---------------------------------------------------------------- invariants

def test_empty_bags_are_exact_zero_for_sum_and_mean():
    tables, ind, off, w = random_problem(2, empty_frac=0.5)
    L = (off[1:] - off[:-1]).numpy()
    for mean in (False, True):
        y = oracle.forward(tables, 9, ind, off, weights=w, mean=mean)
        doff = np.concatenate([[0], np.cumsum([E.shape[1] for E in tables])])
        for t in range(len(tables)):
            for b in range(9):
                if L[t * 9 + b] == 0:
                    assert not y[b, doff[t]:doff[t + 1]].any()
                    assert np.isfinite(y[b, doff[t]:doff[t + 1]]).all()


def test_mean_times_length_equals_sum():
    tables, ind, off, _ = random_problem(4, int_valued=True)
    s = oracle.forward(tables, 9, ind, off)
    m = oracle.forward(tables, 9, ind, off, mean=True)
    L = (off[1:] - off[:-1]).numpy().reshape(len(tables), 9)
    doff = np.concatenate([[0], np.cumsum([E.shape[1] for E in tables])])
    for t in range(len(tables)):
        np.testing.assert_allclose(m[:, doff[t]:doff[t + 1]] * L[t][:, None],
                                   s[:, doff[t]:doff[t + 1]], rtol=1e-14, atol=0)


def test_unit_weights_reproduce_sum_and_linearity_is_exact():
    tables, ind, off, _ = random_problem(8)
    ones = np.ones(ind.numel(), dtype=np.float32)
    s = oracle.forward(tables, 9, ind, off)
    np.testing.assert_array_equal(oracle.forward(tables, 9, ind, off, weights=ones), s)
    doubled = [E * 2 for E in tables]  # exact in fp32
    np.testing.assert_array_equal(oracle.forward(doubled, 9, ind, off), 2 * s)


def test_permuting_within_bags_keeps_output():
    tables, ind, off, _ = random_problem(9, int_valued=True, max_len=20)
    perm_ind = ind.clone()
    g = torch.Generator().manual_seed(1)
    for k in range(off.numel() - 1):
        s, e = int(off[k]), int(off[k + 1])
        perm_ind[s:e] = ind[s:e][torch.randperm(e - s, generator=g)]
    np.testing.assert_array_equal(oracle.forward(tables, 9, perm_ind, off),
                                  oracle.forward(tables, 9, ind, off))


def test_table_blocks_are_independent():
    tables, ind, off, _ = random_problem(10)
    y = oracle.forward(tables, 9, ind, off)
    changed = [tables[0], tables[1] * 0 + 3.0, tables[2]]
    y2 = oracle.forward(changed, 9, ind, off)
    d0, d1 = tables[0].shape[1], tables[1].shape[1]
    np.testing.assert_array_equal(y[:, :d0], y2[:, :d0])
    np.testing.assert_array_equal(y[:, d0 + d1:], y2[:, d0 + d1:])
    assert not np.array_equal(y[:, d0:d0 + d1], y2[:, d0:d0 + d1])


@pytest.mark.parametrize("weighted,mean", [(False, False), (True, True)])
def test_adjoint_identity(weighted, mean):
    # <grad_out, forward(E)> == sum_t <dE_t, E_t>: exact with integer data.
    tables, ind, off, w = random_problem(12, int_valued=True, weighted=weighted, max_len=16)
    rows, dims = table_meta(tables)
    go = torch.randint(-8, 9, (9, int(dims.sum())),
                       generator=torch.Generator().manual_seed(4)).to(torch.float32)
    y = oracle.forward(tables, 9, ind, off, weights=w, mean=mean)
    lhs = float((go.numpy().astype(np.float64) * y).sum())
    res = oracle.backward(rows, dims, 9, ind, off, go, weights=w, mean=mean)
    dense = sparse_to_dense(res, rows, dims)
    rhs = sum(float((d * E.numpy().astype(np.float64)).sum()) for d, E in zip(dense, tables))
    if mean:
        assert lhs == pytest.approx(rhs, rel=1e-13)
    else:
        assert lhs == rhs


def test_sorted_structure_is_a_stable_sort():
    tables, ind, off, _ = random_problem(13, rows=(5, 3, 4), max_len=25)
    rows, dims = table_meta(tables)
    go = torch.zeros(9, int(dims.sum()))
    res = oracle.backward(rows, dims, 9, ind, off, go)
    n = ind.numel()
    assert sorted(res.perm.tolist()) == list(range(n))
    row_base = np.concatenate([[0], np.cumsum(rows)])
    table_of = np.searchsorted(off.numpy()[::9][1:], np.arange(n), side="right")
    key = row_base[table_of] + ind.numpy()
    ks = key[res.perm]
    assert (np.diff(ks) >= 0).all()
    ties = np.diff(ks) == 0
    assert (np.diff(res.perm)[ties] > 0).all()  # equal keys keep ascending positions
    assert (np.diff(res.uniq) > 0).all()
    assert res.seg_start[-1] == n and int(np.diff(res.seg_start).sum()) == n
    np.testing.assert_array_equal(res.uniq, np.unique(key))
    np.testing.assert_array_equal(np.diff(res.seg_start), np.unique(key, return_counts=True)[1])
    for t in range(len(rows) + 1):
        assert res.table_offsets[t] == np.searchsorted(res.uniq, row_base[t])


def test_thread_count_does_not_change_results():
    tables, ind, off, w = random_problem(14, weighted=True, max_len=50)
    a = oracle.forward(tables, 9, ind, off, weights=w, mean=True, threads=1)
    b = oracle.forward(tables, 9, ind, off, weights=w, mean=True, threads=4)
    np.testing.assert_array_equal(a, b)


def test_int32_indices_give_the_same_result():
    tables, ind, off, w = random_problem(15, weighted=True)
    a = oracle.forward(tables, 9, ind, off, weights=w)
    b = oracle.forward(tables, 9, ind.to(torch.int32), off.to(torch.int32), weights=w)
    np.testing.assert_array_equal(a, b)


# ---------------------------------------------------------------- errors

def test_out_of_range_index_is_an_error():
    tables, ind, off, _ = random_problem(16)
    for bad in (-1, tables[0].shape[0]):
        ind2 = ind.clone()
        ind2[int(off[0]):int(off[9])][0:1] = bad
        if int(off[9]) == int(off[0]):
            pytest.skip("first table empty")
        with pytest.raises(oracle.OracleError) as e:
            oracle.forward(tables, 9, ind2, off)
        assert e.value.code == oracle.INDEX_OOB


@pytest.mark.parametrize("mutate", ["first", "decreasing", "last"])
def test_malformed_offsets_are_an_error(mutate):
    tables, ind, off, _ = random_problem(17, empty_frac=0.0)
    off2 = off.clone()
    if mutate == "first":
        off2[0] = 1
    elif mutate == "decreasing":
        off2[5] = off2[4] - 1
    else:
        off2[-1] = off2[-1] - 1
    with pytest.raises(oracle.OracleError) as e:
        oracle.forward(tables, 9, ind, off2)
    assert e.value.code == oracle.BAD_OFFSETS
    rows, dims = table_meta(tables)
    with pytest.raises(oracle.OracleError):
        oracle.backward(rows, dims, 9, ind, off2, torch.zeros(9, int(dims.sum())))


# ---------------------------------------------------------------- weight gradient

@pytest.mark.parametrize("case", ["sum", "mean"])
def test_weight_grad_hand_worked(golden, case):
    g, tables, ind, off, _, go = _golden_problem(golden)
    got = oracle.weight_grad(tables, g["batch"], ind, off, go, mean=case == "mean")
    want = np.array([parse_value(v) for v in g["weight_grad"][case]])
    np.testing.assert_allclose(got, want, rtol=1e-15, atol=0)


@pytest.mark.parametrize("mean", [False, True])
def test_weight_grad_matches_torch_autograd(mean):
    tables, ind, off, w = random_problem(41, weighted=True, max_len=30)
    rows, dims = table_meta(tables)
    go = torch.randn(9, int(dims.sum()), generator=torch.Generator().manual_seed(4),
                     dtype=torch.float32)
    wl_ = w.to(torch.float64).clone().requires_grad_(True)
    y = torch_forward_f64(tables, 9, ind, off, wl_, mean)
    (y * go.to(torch.float64)).sum().backward()
    got = oracle.weight_grad(tables, 9, ind, off, go, mean=mean)
    np.testing.assert_allclose(got, wl_.grad.numpy(), rtol=1e-12, atol=1e-13)


@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
def test_weight_grad_adjoint_identity_and_exact_differences(dtype):
    # y is linear in the weights: <grad_out, y(w)> = sum_i w_i * grad_w_i, and
    # with integer data y(w + e_i) - y(w) gives grad_w_i exactly.
    tables, ind, off, w = random_problem(42, dtype=dtype, int_valued=True, weighted=True,
                                         max_len=20)
    rows, dims = table_meta(tables)
    go = torch.randint(-8, 9, (9, int(dims.sum())),
                       generator=torch.Generator().manual_seed(5)).to(torch.float32)
    gw = oracle.weight_grad(tables, 9, ind, off, go)
    y = oracle.forward(tables, 9, ind, off, weights=w)
    gd = go.double().numpy()
    assert (gd * y).sum() == (w.double().numpy() * gw).sum()
    for i in range(0, ind.numel(), max(1, ind.numel() // 25)):
        w2 = w.clone()
        w2[i] += 1.0
        dy = oracle.forward(tables, 9, ind, off, weights=w2) - y
        assert (gd * dy).sum() == gw[i]
