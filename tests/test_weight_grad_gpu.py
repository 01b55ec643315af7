"""Gradient of the per-sample weights on the GPU (through the C ABI) against the fp64 oracle."""

import numpy as np
import pytest
import torch

import oracle
from tests.conftest import parse_value
from tests.helpers import compact_tables, random_problem
from paper_2609_30656_gb300 import workloads as wl

pytestmark = pytest.mark.gpu
DEV = torch.device("cuda:0")


def _tbe(tables, mean=False, **kw):
    from paper_2609_30656_gb300.tbe import TBE
    return TBE([t.to(DEV).contiguous() for t in tables], pooling="mean" if mean else "sum",
               validate=True, **kw)


def _reference(tables, batch, ind, off, go, mean):
    ref = oracle.weight_grad(tables, batch, ind, off, go, mean=mean)
    scale = oracle.weight_grad([t.abs() for t in tables], batch, ind, off, go.abs(), mean=mean)
    return ref, scale


def _assert_close(got, ref, scale, rtol, what=""):
    got = got.detach().cpu().double().numpy()
    bad = np.abs(got - ref) > rtol * scale + 1e-30
    if bad.any():
        i = int(np.argwhere(bad)[0][0])
        raise AssertionError(f"{what}: {int(bad.sum())} off; first at {i}: gpu {got[i]!r} "
                             f"oracle {ref[i]!r} scale {scale[i]!r}")


@pytest.mark.parametrize("case", ["sum", "mean"])
def test_hand_worked(golden, case):
    g = golden("two_tables_hand.json")
    tables = [torch.tensor(t, dtype=torch.float32) for t in g["tables"]]
    m = _tbe(tables, mean=case == "mean")
    got = m.weight_grad(torch.tensor(g["indices"]).to(DEV), torch.tensor(g["offsets"]).to(DEV),
                        torch.tensor(g["grad_out"], dtype=torch.float32).to(DEV))
    want = np.array([parse_value(v) for v in g["weight_grad"][case]])
    np.testing.assert_allclose(got.cpu().double().numpy(), want, rtol=1e-6, atol=0)
    if case == "sum":
        np.testing.assert_array_equal(got.cpu().double().numpy(), want)


@pytest.mark.parametrize("dtype", [torch.float32, torch.float16, torch.bfloat16])
@pytest.mark.parametrize("mean", [False, True])
def test_random_ragged_within_tolerance(dtype, mean):
    # dims from 8 to 512 (one to four vectors per lane), bags empty to 3000 long
    dims = (8, 64, 128, 256, 512 if dtype != torch.float32 else 96, 12 if dtype == torch.float32 else 24)
    tables, ind, off, _ = random_problem(61, dims=dims, rows=(40, 1000, 5000, 300, 64, 9), batch=33,
                                         max_len=3000, dtype=dtype, empty_frac=0.3)
    go = torch.randn(33, sum(dims), generator=torch.Generator().manual_seed(6))
    m = _tbe(tables, mean=mean)
    got = m.weight_grad(ind.to(DEV), off.to(DEV), go.to(DEV))
    torch.cuda.synchronize()
    ref, scale = _reference(tables, 33, ind, off, go, mean)
    _assert_close(got, ref, scale, 1e-5, f"{dtype} mean={mean}")


@pytest.mark.parametrize("dtype", [torch.float32, torch.float16, torch.bfloat16])
def test_integer_data_bit_exact(dtype):
    tables, ind, off, _ = random_problem(62, dims=(16, 64, 128, 256), rows=(50, 300, 2000, 70),
                                         batch=40, max_len=900, dtype=dtype, int_valued=True)
    go = torch.randint(-8, 9, (40, 464), generator=torch.Generator().manual_seed(7)).float()
    got = _tbe(tables).weight_grad(ind.to(DEV), off.to(DEV), go.to(DEV))
    torch.cuda.synchronize()
    np.testing.assert_array_equal(got.cpu().double().numpy(),
                                  oracle.weight_grad(tables, 40, ind, off, go))


def test_out_of_range_index_gives_zero_and_reports():
    from paper_2609_30656_gb300.tbe import CB_ERR_INDEX_OOB, TBE
    tables, ind, off, _ = random_problem(63, empty_frac=0.0)
    bad = ind.clone()
    bad[3] = 10_000
    go = torch.randn(9, 48)
    m = TBE([t.to(DEV) for t in tables])
    got = m.weight_grad(bad.to(DEV), off.to(DEV), go.to(DEV))
    assert m.get_error() == CB_ERR_INDEX_OOB
    ref, scale = _reference(tables, 9, ind, off, go, False)
    ref[3] = 0.0
    scale[3] = 0.0
    _assert_close(got, ref, scale, 1e-5)


def test_full_size_cfg4_weighted_mean():
    # 64 tables x 1M rows, dims 64/128/256 bf16, batch 8192, lognormal bags,
    # weighted mean: every lookup's weight gradient against the oracle.
    w = wl.get_workload("cfg4")
    tables = wl.make_tables(w, 0, DEV)
    b = wl.make_batch(w, 0, DEV)
    go = wl.make_grad_out(w, 0, DEV)
    m = _tbe(tables, mean=True)
    got = m.weight_grad(b.indices, b.offsets, go)
    torch.cuda.synchronize()
    host_tabs, host_ind = compact_tables(tables, b.indices, b.offsets, w.num_tables, w.batch)
    ref, scale = _reference(host_tabs, w.batch, host_ind, b.offsets.cpu(), go.cpu(), True)
    _assert_close(got, ref, scale, 1e-5, "cfg4")
