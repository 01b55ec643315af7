"""Forward gather-pool on the GPU (through the C ABI) against the fp64 oracle."""

import numpy as np
import pytest
import torch

from tests.conftest import parse_value
from tests.helpers import (RTOL, assert_forward_close, compact_tables, forward_reference,
                           random_problem, sub_batch)
from paper_2609_30656_gb300 import workloads as wl

pytestmark = pytest.mark.gpu
DEV = torch.device("cuda:0")


def _tbe(tables, pooling="sum", index_dtype=torch.int64, **kw):
    from paper_2609_30656_gb300.tbe import TBE
    return TBE([t.to(DEV).contiguous() for t in tables], pooling=pooling,
               index_dtype=index_dtype, validate=True, **kw)


def _run(tables, batch, ind, off, w, mean, index_dtype=torch.int64):
    m = _tbe(tables, "mean" if mean else "sum", index_dtype)
    y = m.forward(ind.to(DEV), off.to(DEV), None if w is None else w.to(DEV))
    torch.cuda.synchronize()
    assert m.get_error() == 0
    return y


@pytest.mark.parametrize("case", ["sum", "mean", "weighted_sum", "weighted_mean"])
def test_hand_worked(golden, case):
    g = golden("two_tables_hand.json")
    tables = [torch.tensor(t, dtype=torch.float32) for t in g["tables"]]
    ind = torch.tensor(g["indices"])
    off = torch.tensor(g["offsets"])
    w = torch.tensor(g["weights"], dtype=torch.float32) if case.startswith("weighted") else None
    y = _run(tables, g["batch"], ind, off, w, case.endswith("mean")).cpu().double().numpy()
    want = np.array([[parse_value(v) for v in row] for row in g["forward"][case]])
    np.testing.assert_allclose(y, want, rtol=1e-6, atol=0)
    if case in ("sum", "weighted_sum"):
        np.testing.assert_array_equal(y, want)  # every value exact in fp32


@pytest.mark.parametrize("dtype", [torch.float32, torch.float16, torch.bfloat16])
@pytest.mark.parametrize("weighted", [False, True])
def test_integer_tables_bit_exact(dtype, weighted):
    # Integer data: every partial sum is exact, so any summation order (including
    # bags split across chunks) must reproduce the oracle bit for bit.
    tables, ind, off, w = random_problem(21, dims=(64, 128, 256, 8), rows=(50, 3000, 17, 9),
                                         batch=40, max_len=1500, dtype=dtype, int_valued=True,
                                         weighted=weighted)
    y = _run(tables, 40, ind, off, w, False)
    ref, _ = forward_reference(tables, 40, ind, off, w, False)
    np.testing.assert_array_equal(y.cpu().double().numpy(), ref)


@pytest.mark.parametrize("dtype", [torch.float32, torch.float16, torch.bfloat16])
@pytest.mark.parametrize("weighted,mean", [(False, False), (False, True), (True, False),
                                           (True, True)])
def test_random_ragged_within_tolerance(dtype, weighted, mean):
    # Ragged bags from empty to 3000 long (several 512-lookup chunks), mixed dims.
    tables, ind, off, w = random_problem(22, dims=(8, 64, 128, 256, 512 if dtype != torch.float32 else 96),
                                         rows=(40, 1000, 5000, 300, 64), batch=33, max_len=3000,
                                         dtype=dtype, weighted=weighted, empty_frac=0.3)
    y = _run(tables, 33, ind, off, w, mean)
    ref, scale = forward_reference(tables, 33, ind, off, w, mean)
    assert_forward_close(y, ref, scale, RTOL[dtype], f"{dtype} w={weighted} mean={mean}")


def test_row_sizes_not_a_power_of_two_vectors():
    # 48-byte and 384-byte rows (3 and 24 vectors) take the one-row-per-step path.
    tables, ind, off, w = random_problem(23, dims=(12, 96, 24), rows=(100, 100, 100), batch=20,
                                         max_len=700, dtype=torch.float32)
    tables[2] = tables[2].to(torch.float16)
    y = _run(tables, 20, ind, off, w, False)
    ref, scale = forward_reference(tables, 20, ind, off, w, False)
    assert_forward_close(y, ref, scale, 2e-3)


def test_int32_indices_and_offsets():
    tables, ind, off, w = random_problem(24, batch=50, max_len=900, weighted=True)
    y = _run(tables, 50, ind.to(torch.int32), off.to(torch.int32), w, True,
             index_dtype=torch.int32)
    ref, scale = forward_reference(tables, 50, ind, off, w, True)
    assert_forward_close(y, ref, scale, 1e-5)


def test_all_bags_empty_and_single_lookup_bags():
    tables, _, _, _ = random_problem(25)
    off = torch.zeros(3 * 9 + 1, dtype=torch.int64)
    y = _run(tables, 9, torch.zeros(0, dtype=torch.int64), off, None, True)
    assert (y == 0).all()
    # one-hot bags
    off = torch.arange(3 * 9 + 1, dtype=torch.int64)
    ind = torch.cat([torch.randint(0, r, (9,)) for r in (7, 50, 13)])
    y = _run(tables, 9, ind, off, None, False)
    ref, scale = forward_reference(tables, 9, ind, off, None, False)
    assert_forward_close(y, ref, scale, 1e-5)


def test_bitwise_deterministic():
    tables, ind, off, w = random_problem(26, batch=64, max_len=2000, weighted=True)
    a = _run(tables, 64, ind, off, w, True)
    b = _run(tables, 64, ind, off, w, True)
    assert torch.equal(a, b)


def test_out_of_range_index_reports_and_contributes_nothing():
    from paper_2609_30656_gb300.tbe import CB_ERR_INDEX_OOB, CbTbeError
    tables, ind, off, _ = random_problem(27, empty_frac=0.0)
    bad = ind.clone()
    bad[0] = 10_000
    m = _tbe(tables)
    with pytest.raises(CbTbeError) as e:
        m.forward(bad.to(DEV), off.to(DEV))
    assert e.value.status == CB_ERR_INDEX_OOB
    # without validation the error is sticky until read
    from paper_2609_30656_gb300.tbe import TBE
    m2 = TBE([t.to(DEV) for t in tables])
    y = m2.forward(bad.to(DEV), off.to(DEV))
    assert m2.get_error() == CB_ERR_INDEX_OOB
    assert m2.get_error() == 0
    zeroed = ind.clone()
    ref_tables = [t.clone() for t in tables]
    # the bad lookup contributes nothing: same as the bag without that lookup
    ref_tables[0] = torch.cat([ref_tables[0], torch.zeros(1, ref_tables[0].shape[1])])
    zeroed[0] = ref_tables[0].shape[0] - 1
    ref, scale = forward_reference(ref_tables, 9, zeroed, off, None, False)
    assert_forward_close(y, ref, scale, 1e-5)


@pytest.mark.parametrize("mutate", ["first", "decreasing", "last"])
def test_malformed_offsets_report(mutate):
    from paper_2609_30656_gb300.tbe import CB_ERR_BAD_OFFSETS, CbTbeError
    tables, ind, off, _ = random_problem(28, empty_frac=0.0)
    off2 = off.clone()
    if mutate == "first":
        off2[0] = 1
    elif mutate == "decreasing":
        off2[5] = off2[4] - 1
    else:
        off2[-1] = off2[-1] - 1
    m = _tbe(tables)
    with pytest.raises(CbTbeError) as e:
        m.forward(ind.to(DEV), off2.to(DEV))
    assert e.value.status == CB_ERR_BAD_OFFSETS


# ----------------------------------------------------------------------------- workloads

def _workload_forward(name, cols=None, seed=0):
    w = wl.get_workload(name)
    tables = wl.make_tables(w, seed, DEV)
    b = wl.make_batch(w, seed, DEV)
    from paper_2609_30656_gb300.tbe import TBE
    m = TBE(tables, pooling="mean" if w.mean else "sum", validate=True)
    y = m.forward(b.indices, b.offsets, b.weights)
    torch.cuda.synchronize()
    if cols is None:
        host_tabs, host_ind = compact_tables(tables, b.indices, b.offsets, w.num_tables, w.batch)
        ref, scale = forward_reference(host_tabs, w.batch, host_ind, b.offsets.cpu(),
                                       None if b.weights is None else b.weights.cpu(), w.mean)
        assert_forward_close(y, ref, scale, RTOL[w.torch_dtype], name)
    else:
        ind, off, wt = sub_batch(b.indices, b.offsets, b.weights, w.num_tables, w.batch, cols)
        host_tabs, host_ind = compact_tables(tables, ind.to(DEV), off, w.num_tables, len(cols))
        ref, scale = forward_reference(host_tabs, len(cols), host_ind, off, wt, w.mean)
        assert_forward_close(y[torch.as_tensor(cols, device=DEV)], ref, scale,
                             RTOL[w.torch_dtype], name)
    return w, b


@pytest.mark.parametrize("name", ["cfg1", "cfg2", "cfg3", "cfg4"])
def test_workload_full_size(name):
    _workload_forward(name)


@pytest.mark.slow
@pytest.mark.parametrize("name", ["cfg5", "cfg5u"])
def test_cfg5_full_size_sampled_rows(name):
    # 128 GB of tables: every output row b of a sample of batch rows, including
    # the rows that hold the longest bags, is checked element by element.
    w = wl.get_workload(name)
    g = torch.Generator().manual_seed(7)
    b_probe = wl.make_batch(w, 0, DEV)
    L = (b_probe.offsets[1:] - b_probe.offsets[:-1]).view(w.num_tables, w.batch)
    heavy = torch.unique(L.argmax(dim=1)).cpu()[:16]
    cols = torch.unique(torch.cat([heavy, torch.randint(0, w.batch, (48,), generator=g)]))
    del b_probe
    _workload_forward(name, cols=cols.tolist())
