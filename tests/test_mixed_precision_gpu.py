"""Mixed precision on the GPU (CB_OUT_F16 / CB_OUT_BF16): the pooled output in
fp16 / bf16 and grad_out in the same type, against the fp64 oracle. The oracle
reads grad_out's stored values exactly (widened), so the backward keeps the
fp32 bound; the forward adds one rounding of the output type."""

import numpy as np
import pytest
import torch

import oracle
from tests.helpers import (RTOL, RTOL_BWD, assert_backward_matches, backward_reference,
                           forward_reference, random_problem, table_meta)

pytestmark = pytest.mark.gpu
DEV = torch.device("cuda:0")
OUT = [torch.float16, torch.bfloat16]
DIMS = (8, 64, 128, 256, 512)
ROWS = (40, 1000, 5000, 300, 64)


def _ulp(x, dtype):
    mant, emin = {torch.float16: (10, -14), torch.bfloat16: (7, -126)}[dtype]
    e = np.floor(np.log2(np.maximum(np.abs(x), 2.0 ** emin)))
    return 2.0 ** (e - mant)


def _tbe(tables, out_dtype, mean=False):
    from paper_2609_30656_gb300.tbe import TBE
    return TBE([t.to(DEV).contiguous() for t in tables], pooling="mean" if mean else "sum",
               validate=True, out_dtype=out_dtype)


@pytest.mark.parametrize("out_dtype", OUT)
@pytest.mark.parametrize("dtype", [torch.float32, torch.float16, torch.bfloat16])
@pytest.mark.parametrize("weighted,mean", [(False, False), (True, True)])
def test_forward_half_output_within_tolerance(out_dtype, dtype, weighted, mean):
    tables, ind, off, w = random_problem(111, dims=DIMS, rows=ROWS, batch=33, max_len=3000, dtype=dtype,
                                         weighted=weighted, empty_frac=0.3)
    m = _tbe(tables, out_dtype, mean)
    y = m.forward(ind.to(DEV), off.to(DEV), None if w is None else w.to(DEV))
    torch.cuda.synchronize()
    assert y.dtype == out_dtype
    ref, scale = forward_reference(tables, 33, ind, off, w, mean)
    got = y.cpu().double().numpy()
    bad = np.abs(got - ref) > RTOL[dtype] * scale + _ulp(ref, out_dtype) + 1e-30
    assert not bad.any(), (np.argwhere(bad)[:3], got[bad][:3], ref[bad][:3])


@pytest.mark.parametrize("out_dtype", OUT)
def test_integer_data_bit_exact(out_dtype):
    # sums of at most 20 integers in [-8, 8] are exact in fp16 and bf16
    tables, ind, off, w = random_problem(112, dims=(16, 128), rows=(50, 3000), batch=40, max_len=20,
                                         int_valued=True, dtype=torch.bfloat16)
    m = _tbe(tables, out_dtype)
    y = m.forward(ind.to(DEV), off.to(DEV))
    ref, _ = forward_reference(tables, 40, ind, off, None, False)
    np.testing.assert_array_equal(y.cpu().double().numpy(), ref)
    rows, dims = table_meta(tables)
    go = torch.randint(-8, 9, (40, int(dims.sum())), generator=torch.Generator().manual_seed(4)).to(out_dtype)
    g = m.backward(ind.to(DEV), off.to(DEV), go.to(DEV))
    torch.cuda.synchronize()
    res, sc = backward_reference(rows, dims, 40, ind, off, go.float(), None, False)
    assert_backward_matches(g, res, sc, rtol=0.0)


@pytest.mark.parametrize("out_dtype", OUT)
@pytest.mark.parametrize("weighted,mean", [(False, False), (True, True)])
def test_backward_half_grad_out_within_tolerance(out_dtype, weighted, mean):
    tables, ind, off, w = random_problem(113, dims=DIMS, rows=ROWS, batch=37, max_len=900,
                                         dtype=torch.float16, weighted=weighted, empty_frac=0.3)
    rows, dims = table_meta(tables)
    go = torch.randn(37, int(dims.sum()), generator=torch.Generator().manual_seed(5)).to(out_dtype)
    m = _tbe(tables, out_dtype, mean)
    g = m.backward(ind.to(DEV), off.to(DEV), go.to(DEV), None if w is None else w.to(DEV))
    torch.cuda.synchronize()
    res, sc = backward_reference(rows, dims, 37, ind, off, go.float(), w, mean)
    assert_backward_matches(g, res, sc, rtol=RTOL_BWD, what=f"{out_dtype}")


@pytest.mark.parametrize("out_dtype", OUT)
def test_weight_grad_and_fused_step_with_half_grad_out(out_dtype):
    tables, ind, off, w = random_problem(114, dims=(8, 64, 128), rows=(20, 300, 3000), batch=30,
                                         max_len=600, weighted=True)
    rows, dims = table_meta(tables)
    go = torch.randn(30, int(dims.sum()), generator=torch.Generator().manual_seed(6)).to(out_dtype)
    m = _tbe(tables, out_dtype, mean=True)
    gw = m.weight_grad(ind.to(DEV), off.to(DEV), go.to(DEV))
    torch.cuda.synchronize()
    ref = oracle.weight_grad(tables, 30, ind, off, go.float(), mean=True)
    scale = oracle.weight_grad([t.abs() for t in tables], 30, ind, off, go.float().abs(), mean=True)
    assert (np.abs(gw.cpu().double().numpy() - ref) <= 1e-5 * scale + 1e-30).all()
    # fused SGD with lr = 1/8 on the same inputs
    m.backward_apply(ind.to(DEV), off.to(DEV), go.to(DEV), w.to(DEV), optimizer="sgd", lr=0.125)
    torch.cuda.synchronize()
    want, _ = oracle.apply_step(tables, 30, ind, off, go.float(), weights=w, mean=True, kind="sgd", lr=0.125)
    _, sg = backward_reference(rows, dims, 30, ind, off, go.float(), w, True)
    tol_abs = 0.125 * 2e-5 * sg.max() + 1e-6 * max(float(t.abs().max()) for t in tables)
    for t0, t1 in zip(m.tables, want):
        assert (np.abs(t0.cpu().double().numpy() - t1.double().numpy()) <= tol_abs).all()


def test_dims_not_a_multiple_of_8_are_rejected_for_half_output():
    from paper_2609_30656_gb300.tbe import CbTbeError, TBE
    t = torch.zeros(10, 4, device=DEV)  # 16-byte fp32 rows, but 8-byte fp16 grad_out rows
    with pytest.raises(CbTbeError):
        TBE([t], out_dtype=torch.float16)
    TBE([t])  # fine with fp32 output
