"""Factorization-machine cross term on the GPU (through the C ABI) against the fp64 oracle."""

import numpy as np
import pytest
import torch

import oracle
from tests.helpers import forward_reference
from paper_2609_30656_gb300 import workloads as wl

pytestmark = pytest.mark.gpu
DEV = torch.device("cuda:0")
U32 = 2.0 ** -24  # unit roundoff of fp32


def _fm_rtol(T):
    # Column sums of T terms (sequential per lane, then a butterfly over field
    # groups), a square, a subtraction and a sum over at most 512 columns:
    # a bound of (3 (T + 5) + 40) u relative to 1/2 sum_j (sum_t |v_tj|)^2.
    return (3 * (T + 5) + 40) * U32


def _fm_scale(y, T):
    B = y.shape[0]
    a = np.abs(y.astype(np.float64)).reshape(B, T, -1)
    return 0.5 * (a.sum(1) ** 2).sum(-1)


def _check_fm(y_dev, T, g_dev=None):
    from paper_2609_30656_gb300 import tbe
    y = y_dev.cpu().numpy()
    got = tbe.fm_forward(y_dev, T).cpu().double().numpy()
    torch.cuda.synchronize()
    want = oracle.fm_forward(y, T)
    bad = np.abs(got - want) > _fm_rtol(T) * _fm_scale(y, T) + 1e-30
    assert not bad.any(), f"fm off at {np.argwhere(bad)[:3].ravel()}"
    if g_dev is not None:
        gy = tbe.fm_backward(y_dev, g_dev, T).cpu().double().numpy()
        gw = oracle.fm_backward(y, g_dev.cpu().numpy(), T)
        B = y.shape[0]
        colsum = np.abs(y.astype(np.float64)).reshape(B, T, -1).sum(1, keepdims=True)
        sc = (np.abs(g_dev.cpu().double().numpy())[:, None, None] * colsum).repeat(T, 1).reshape(B, -1)
        bad = np.abs(gy - gw) > (T + 8) * U32 * sc + 1e-30
        assert not bad.any(), f"grad off at {np.argwhere(bad)[:3].ravel()}"


@pytest.mark.parametrize("D", [4, 8, 16, 32, 64, 128, 256, 384, 512, 12, 96, 200])
@pytest.mark.parametrize("T", [1, 2, 3, 26])
def test_every_field_layout_within_tolerance(D, T):
    g = torch.Generator(device=DEV).manual_seed(D * 100 + T)
    B = 37
    y = torch.randn(B, T * D, generator=g, device=DEV)
    _check_fm(y, T, torch.randn(B, generator=g, device=DEV))


def test_integer_inputs_bit_exact():
    from paper_2609_30656_gb300 import tbe
    g = torch.Generator(device=DEV).manual_seed(7)
    for T, D in [(26, 16), (7, 64), (3, 128)]:
        y = torch.randint(-4, 5, (50, T * D), generator=g, device=DEV).float()
        gf = torch.randint(-3, 4, (50,), generator=g, device=DEV).float()
        np.testing.assert_array_equal(tbe.fm_forward(y, T).cpu().double().numpy(),
                                      oracle.fm_forward(y.cpu().numpy(), T))
        np.testing.assert_array_equal(tbe.fm_backward(y, gf, T).cpu().double().numpy(),
                                      oracle.fm_backward(y.cpu().numpy(), gf.cpu().numpy(), T))


def test_row_stride_and_untouched_columns():
    from paper_2609_30656_gb300 import tbe
    g = torch.Generator(device=DEV).manual_seed(8)
    T, D, B = 5, 32, 20
    wide = torch.randn(B, T * D + 16, generator=g, device=DEV)
    y = wide[:, :T * D]
    gf = torch.randn(B, generator=g, device=DEV)
    _check_fm(y, T, gf)
    out = torch.full_like(wide, 7.0)
    tbe.fm_backward(y, gf, T, out=out[:, :T * D])
    assert (out[:, T * D:] == 7.0).all()


def test_empty_batch_and_bad_arguments():
    from paper_2609_30656_gb300 import tbe
    assert tbe.fm_forward(torch.zeros(0, 64, device=DEV), 2).numel() == 0
    with pytest.raises(tbe.CbTbeError):
        tbe.fm_forward(torch.zeros(3, 18, device=DEV), 3)  # dim 6 is not a multiple of 4


def test_full_size_cfg5_layout_sampled_rows():
    # The pooled output of cfg5: 65536 samples x 100 fields x 128 columns.
    from paper_2609_30656_gb300 import tbe
    g = torch.Generator(device=DEV).manual_seed(9)
    B, T, D = 65536, 100, 128
    y = torch.randn(B, T * D, generator=g, device=DEV) * 0.05
    gf = torch.randn(B, generator=g, device=DEV)
    fm = tbe.fm_forward(y, T)
    gy = tbe.fm_backward(y, gf, T)
    torch.cuda.synchronize()
    rows = torch.randint(0, B, (96,), generator=torch.Generator().manual_seed(1))
    rows = torch.cat([rows, torch.tensor([0, B - 1])])
    ys = y[rows.to(DEV)].cpu().numpy()
    want = oracle.fm_forward(ys, T)
    assert (np.abs(fm[rows.to(DEV)].cpu().double().numpy() - want)
            <= _fm_rtol(T) * _fm_scale(ys, T)).all()
    gw = oracle.fm_backward(ys, gf[rows.to(DEV)].cpu().numpy(), T)
    colsum = np.abs(ys.astype(np.float64)).reshape(len(rows), T, D).sum(1, keepdims=True)
    sc = (np.abs(gf[rows.to(DEV)].cpu().double().numpy())[:, None, None] * colsum).repeat(T, 1)
    assert (np.abs(gy[rows.to(DEV)].cpu().double().numpy() - gw)
            <= (T + 8) * U32 * sc.reshape(len(rows), -1)).all()


def test_on_the_pooled_output_of_cfg3():
    # The lookup of the 26-feature CTR-benchmark shape followed by the FM term,
    # against the oracle's lookup followed by the oracle's FM term.
    from paper_2609_30656_gb300 import tbe
    w = wl.get_workload("cfg3")
    tables = wl.make_tables(w, 0, DEV)
    b = wl.make_batch(w, 0, DEV)
    m = tbe.TBE(tables, validate=True)
    y = m.forward(b.indices, b.offsets)
    fm = tbe.fm_forward(y, w.num_tables)
    torch.cuda.synchronize()
    ref_y, _ = forward_reference([t.cpu() for t in tables], w.batch, b.indices.cpu(),
                                 b.offsets.cpu(), None, False)
    want = oracle.fm_forward(ref_y.astype(np.float32), w.num_tables)
    # y itself differs from the fp64 pooled rows by its fp32 rounding (and the
    # fp16 tables' sums), so compare with the FM bound plus that rounding.
    scale = _fm_scale(ref_y.astype(np.float32), w.num_tables)
    assert (np.abs(fm.cpu().double().numpy() - want) <= (_fm_rtol(w.num_tables) + 4 * U32) * scale).all()
