"""De-duplicated backward on the GPU (through the C ABI) against the fp64 oracle."""

import numpy as np
import pytest
import torch

from tests.conftest import parse_value
from tests.helpers import (assert_backward_matches, backward_reference, random_problem,
                           table_meta)
from paper_2609_30656_gb300 import workloads as wl

pytestmark = pytest.mark.gpu
DEV = torch.device("cuda:0")


def _tbe(tables, pooling="sum", index_dtype=torch.int64, validate=True, **kw):
    from paper_2609_30656_gb300.tbe import TBE
    return TBE([t.to(DEV).contiguous() for t in tables], pooling=pooling,
               index_dtype=index_dtype, validate=validate, **kw)


def _run(tables, batch, ind, off, go, w, mean, index_dtype=torch.int64):
    m = _tbe(tables, "mean" if mean else "sum", index_dtype)
    g = m.backward(ind.to(DEV), off.to(DEV), go.to(DEV), None if w is None else w.to(DEV))
    torch.cuda.synchronize()
    return g


@pytest.mark.parametrize("case", ["sum", "weighted_mean"])
def test_hand_worked(golden, case):
    gd = golden("two_tables_hand.json")
    tables = [torch.tensor(t, dtype=torch.float32) for t in gd["tables"]]
    ind = torch.tensor(gd["indices"])
    off = torch.tensor(gd["offsets"])
    go = torch.tensor(gd["grad_out"], dtype=torch.float32)
    w = torch.tensor(gd["weights"], dtype=torch.float32) if case == "weighted_mean" else None
    g = _run(tables, gd["batch"], ind, off, go, w, case == "weighted_mean")
    b = gd["backward"]
    U = g.num_unique
    assert g.unique_ids[:U].tolist() == b["uniq"]
    assert g.table_offsets.tolist() == b["table_offsets"]
    assert g.grad_offsets[:U + 1].tolist() == b["grad_offsets"]
    got = g.grads[:g.num_floats].cpu().double().numpy()
    want = np.array([parse_value(v) for v in b[case]])
    np.testing.assert_allclose(got, want, rtol=1e-6, atol=1e-7)
    if case == "sum":
        np.testing.assert_array_equal(got, want)


@pytest.mark.parametrize("weighted", [False, True])
def test_integer_data_bit_exact(weighted):
    # Few rows, long bags: every row repeats thousands of times, so runs span many
    # 512-position chunks and exercise the fix-up; integer data make it exact.
    tables, ind, off, w = random_problem(31, dims=(64, 128, 8), rows=(3, 40, 2000), batch=50,
                                         max_len=600, int_valued=True, weighted=weighted)
    rows, dims = table_meta(tables)
    go = torch.randint(-8, 9, (50, int(dims.sum())),
                       generator=torch.Generator().manual_seed(1)).to(torch.float32)
    g = _run(tables, 50, ind, off, go, w, False)
    res, scale = backward_reference(rows, dims, 50, ind, off, go, w, False)
    assert_backward_matches(g, res, scale, rtol=0.0)


@pytest.mark.parametrize("weighted,mean", [(False, False), (False, True), (True, False),
                                           (True, True)])
@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
def test_random_within_tolerance(weighted, mean, dtype):
    tables, ind, off, w = random_problem(32, dims=(8, 64, 128, 256, 512), rows=(5, 100, 1000, 64, 7),
                                         batch=37, max_len=900, dtype=dtype, weighted=weighted,
                                         empty_frac=0.3)
    rows, dims = table_meta(tables)
    go = torch.randn(37, int(dims.sum()), generator=torch.Generator().manual_seed(2))
    g = _run(tables, 37, ind, off, go, w, mean)
    res, scale = backward_reference(rows, dims, 37, ind, off, go, w, mean)
    assert_backward_matches(g, res, scale, what=f"w={weighted} mean={mean}")


def test_int32_indices():
    tables, ind, off, w = random_problem(33, batch=30, max_len=400)
    rows, dims = table_meta(tables)
    go = torch.randn(30, int(dims.sum()), generator=torch.Generator().manual_seed(3))
    g = _run(tables, 30, ind.to(torch.int32), off.to(torch.int32), go, w, False,
             index_dtype=torch.int32)
    res, scale = backward_reference(rows, dims, 30, ind, off, go, w, False)
    assert_backward_matches(g, res, scale)


def test_size_query_and_capacity_error():
    from paper_2609_30656_gb300.tbe import CB_ERR_CAPACITY, CbTbeError
    tables, ind, off, w = random_problem(34, batch=20, max_len=50)
    rows, dims = table_meta(tables)
    go = torch.randn(20, int(dims.sum()))
    m = _tbe(tables)
    probe = m.alloc_grad(0, 0, size_only=True)
    m.backward_into(probe, ind.to(DEV), off.to(DEV), go.to(DEV))
    res = backward_reference(rows, dims, 20, ind, off, go, None, False)[0]
    assert probe.num_unique == res.num_unique
    assert probe.num_floats == int(res.grad_offsets[-1])
    small = m.alloc_grad(res.num_unique - 1, int(res.grad_offsets[-1]))
    with pytest.raises(CbTbeError) as e:
        m.backward_into(small, ind.to(DEV), off.to(DEV), go.to(DEV))
    assert e.value.status == CB_ERR_CAPACITY
    assert small.num_unique == res.num_unique  # sizes are still reported


def test_bitwise_deterministic():
    tables, ind, off, w = random_problem(35, rows=(3, 30, 300), batch=64, max_len=800,
                                         weighted=True)
    rows, dims = table_meta(tables)
    go = torch.randn(64, int(dims.sum()))
    a = _run(tables, 64, ind, off, go, w, True)
    b = _run(tables, 64, ind, off, go, w, True)
    assert torch.equal(a.grads[:a.num_floats], b.grads[:b.num_floats])
    assert torch.equal(a.unique_ids[:a.num_unique], b.unique_ids[:b.num_unique])


@pytest.mark.parametrize("weighted,mean", [(False, False), (True, True)])
def test_both_radix_pass_forms_give_the_same_bits(weighted, mean):
    # Reduce-then-scan and single-sweep passes are both stable sorts of the
    # same pairs: the sorted order, and so every gradient bit, must agree.
    # Rows > 2^16 (three passes), hot rows (Zipf) and tables of 1-2 tiles.
    from paper_2609_30656_gb300.tbe import CB_SORT_LOOKBACK
    tables, ind, off, w = random_problem(37, dims=(16, 64, 128), rows=(3, 70000, 300000), batch=700,
                                         max_len=120, weighted=weighted, empty_frac=0.1)
    rows, dims = table_meta(tables)
    go = torch.randn(700, int(dims.sum()), generator=torch.Generator().manual_seed(38))
    args = (ind.to(DEV), off.to(DEV), go.to(DEV), None if w is None else w.to(DEV))
    pooling = "mean" if mean else "sum"
    a = _tbe(tables, pooling).backward(*args)
    b = _tbe(tables, pooling, extra_flags=CB_SORT_LOOKBACK).backward(*args)
    torch.cuda.synchronize()
    assert a.num_unique == b.num_unique and a.num_floats == b.num_floats
    assert torch.equal(a.unique_ids[:a.num_unique], b.unique_ids[:b.num_unique])
    assert torch.equal(a.grads[:a.num_floats], b.grads[:b.num_floats])
    res, scale = backward_reference(rows, dims, 700, ind, off, go, w, mean)
    assert_backward_matches(a, res, scale)


def test_one_table_of_many_radix_tiles():
    # ~4M lookups of one table: ~1000 radix tiles, so the slot scan cuts the
    # table into dozens of segments; both pass forms and the oracle agree.
    from paper_2609_30656_gb300.tbe import CB_SORT_LOOKBACK
    g = torch.Generator().manual_seed(39)
    rows, batch = 200000, 20000
    table = (torch.randn(rows, 16, generator=g) * 0.01).float()
    lens = torch.randint(0, 401, (batch,), generator=g)
    off = torch.zeros(batch + 1, dtype=torch.int64)
    off[1:] = torch.cumsum(lens, 0)
    ind = torch.randint(0, rows, (int(off[-1]),), generator=g)
    go = torch.randn(batch, 16, generator=g)
    args = (ind.to(DEV), off.to(DEV), go.to(DEV))
    a = _tbe([table]).backward(*args)
    b = _tbe([table], extra_flags=CB_SORT_LOOKBACK).backward(*args)
    torch.cuda.synchronize()
    assert ind.numel() > 1000 * 4096 * 0.9
    assert torch.equal(a.unique_ids[:a.num_unique], b.unique_ids[:b.num_unique])
    assert torch.equal(a.grads[:a.num_floats], b.grads[:b.num_floats])
    res, scale = backward_reference(np.array([rows]), np.array([16]), batch, ind, off, go, None, False)
    assert_backward_matches(a, res, scale)


def test_forced_lookback_timeout_returns_an_error_and_the_context_survives():
    from paper_2609_30656_gb300.tbe import CB_DEBUG_FORCE_LOOKBACK_TIMEOUT, CB_ERR_TIMEOUT
    # Enough lookups for several radix tiles; tile 1 waits on a word nothing writes.
    tables, ind, off, _ = random_problem(36, rows=(1000, 1000, 1000), batch=400, max_len=60)
    rows, dims = table_meta(tables)
    go = torch.randn(400, int(dims.sum()))
    m = _tbe(tables, validate=False, extra_flags=CB_DEBUG_FORCE_LOOKBACK_TIMEOUT)
    g = m.alloc_grad(ind.numel(), ind.numel() * int(dims.max()))
    m.backward_into(g, ind.to(DEV), off.to(DEV), go.to(DEV))
    assert m.get_error() == CB_ERR_TIMEOUT
    # the device is still usable afterwards
    g2 = _run(tables, 400, ind, off, go, None, False)
    res, scale = backward_reference(rows, dims, 400, ind, off, go, None, False)
    assert_backward_matches(g2, res, scale)


# ----------------------------------------------------------------------------- workloads

@pytest.mark.parametrize("name", ["cfg2", "cfg3", "cfg4"])
def test_workload_full_size(name):
    w = wl.get_workload(name)
    tables = wl.make_tables(w, 0, DEV)
    b = wl.make_batch(w, 0, DEV)
    go = wl.make_grad_out(w, 0, DEV)
    m = _tbe(tables, "mean" if w.mean else "sum")
    g = m.backward(b.indices, b.offsets, go, b.weights)
    torch.cuda.synchronize()
    rows = np.array(w.rows, np.int64)
    dims = np.array(w.dims, np.int32)
    res, scale = backward_reference(rows, dims, w.batch, b.indices.cpu(), b.offsets.cpu(), go.cpu(),
                                    None if b.weights is None else b.weights.cpu(), w.mean)
    assert_backward_matches(g, res, scale, what=name)


@pytest.mark.slow
@pytest.mark.parametrize("name", ["cfg5", "cfg5u"])
def test_cfg5_full_size_sampled_tables(name):
    # Full 100-table batch on the GPU; three tables (first, middle, last) are
    # checked completely against the oracle run on that table's lookups alone.
    # cfg5u (uniform indices) is the reuse-free control: ~1.7e8 distinct rows,
    # nearly every 32-lookup batch of the reduce holds run ends.
    w = wl.get_workload(name)
    tables = wl.make_tables(w, 0, DEV)
    b = wl.make_batch(w, 0, DEV)
    go = wl.make_grad_out(w, 0, DEV)
    m = _tbe(tables)
    g = m.backward(b.indices, b.offsets, go, b.weights)
    torch.cuda.synchronize()
    U = g.num_unique
    ids = g.unique_ids[:U]
    assert bool((ids[1:] > ids[:-1]).all())
    toff = g.table_offsets.cpu().numpy()
    assert toff[0] == 0 and toff[-1] == U and (np.diff(toff) >= 0).all()
    off = b.offsets.cpu()
    B = w.batch
    for t in (0, w.num_tables // 2, w.num_tables - 1):
        s, e = int(off[t * B]), int(off[(t + 1) * B])
        ind_t = b.indices[s:e].cpu()
        off_t = off[t * B:(t + 1) * B + 1] - s
        go_t = go[:, 128 * t:128 * (t + 1)].cpu().contiguous()
        res, scale = backward_reference(np.array([w.rows[t]]), np.array([128], np.int32), B, ind_t,
                                        off_t, go_t, None, False)
        u0, u1 = int(toff[t]), int(toff[t + 1])
        assert u1 - u0 == res.num_unique
        row_base = t * w.rows[0]
        np.testing.assert_array_equal(ids[u0:u1].cpu().numpy() - row_base, res.uniq)
        f0 = int(g.grad_offsets[u0])
        got = g.grads[f0:f0 + (u1 - u0) * 128].cpu().double().numpy()
        err = np.abs(got - res.grads)
        assert (err <= 1e-5 * scale + 1e-30).all(), f"table {t}: max err {err.max()}"
