"""Segment structures that stress the walkers' batch and window logic, per row layout.

Every compiled row layout (1, 2, 4 or 8 rows per warp step, one 16-byte vector per
lane) is run on bag and run patterns chosen to land on the edges of 32-lookup
batches and 512-lookup chunks: long stretches of empty bags, one-hot bags,
bags ending exactly on a batch edge, bags split across chunks, trailing empty
bags, a table with no lookups, rows repeated thousands of times. Integer data
make every sum exact, so the GPU must match the fp64 oracle bit for bit.
"""

import numpy as np
import pytest
import torch

from tests.helpers import backward_reference, forward_reference, table_meta

pytestmark = pytest.mark.gpu
DEV = torch.device("cuda:0")

# (storage dtype, dim) -> rows per warp step of the forward gather
FWD_LAYOUTS = [
    (torch.float32, 128), (torch.float32, 64), (torch.float32, 32), (torch.float32, 16),
    (torch.float16, 256), (torch.float16, 128), (torch.float16, 64), (torch.float16, 32),
    (torch.bfloat16, 128), (torch.bfloat16, 16),
]
# fp32 gradient rows of dim 128, 64, 32, 16: 1, 2, 4, 8 rows per warp step
BWD_DIMS = [128, 64, 32, 16]


def _lengths(batch: int, g: torch.Generator) -> list[int]:
    """Bag lengths for one table: runs of empties, one-hot bags, batch-edge bags, heavy bags."""
    pattern = ([0] * 70 + [1] * 40 + [32, 32, 31, 33, 1, 0, 0, 64, 5, 27]
               + [700, 0, 3000, 1, 0, 511, 513, 2, 0] + [0] * 35)
    out = list(pattern)
    while len(out) < batch - 40:
        out.append(int(torch.randint(0, 40, (1,), generator=g)))
    out = out[:batch - 40] + [0] * 40  # trailing empty bags: owned by the table's last chunk
    return out


def _problem(dims, dtype, batch, seed, empty_table=True, weighted=False):
    g = torch.Generator().manual_seed(seed)
    rows = [997 + 13 * t for t in range(len(dims))]
    tables = [torch.randint(-8, 9, (r, d), generator=g).to(torch.float32).to(dtype)
              for r, d in zip(rows, dims)]
    lens = []
    for t in range(len(dims)):
        if empty_table and t == 1:
            lens += [0] * batch
        else:
            lens += _lengths(batch, g)
    off = torch.zeros(len(lens) + 1, dtype=torch.int64)
    off[1:] = torch.cumsum(torch.tensor(lens, dtype=torch.int64), 0)
    ind = []
    for t, r in enumerate(rows):
        s, e = int(off[t * batch]), int(off[(t + 1) * batch])
        ind.append(torch.randint(0, r, (e - s,), generator=g))
    ind = torch.cat(ind)
    w = torch.randint(0, 3, (ind.numel(),), generator=g).to(torch.float32) if weighted else None
    return tables, ind, off, w


def _tbe(tables, pooling="sum", validate=True):
    from paper_2609_30656_gb300.tbe import TBE
    return TBE([t.to(DEV).contiguous() for t in tables], pooling=pooling, validate=validate)


@pytest.mark.parametrize("dtype,dim", FWD_LAYOUTS)
@pytest.mark.parametrize("weighted", [False, True])
def test_forward_segment_edges_bit_exact(dtype, dim, weighted):
    batch = 260
    tables, ind, off, w = _problem((dim, dim, dim), dtype, batch, seed=dim + int(weighted),
                                   weighted=weighted)
    m = _tbe(tables)
    y = m.forward(ind.to(DEV), off.to(DEV), None if w is None else w.to(DEV))
    torch.cuda.synchronize()
    ref, _ = forward_reference(tables, batch, ind, off, w, False)
    np.testing.assert_array_equal(y.cpu().double().numpy(), ref)


@pytest.mark.parametrize("dtype,dim", [(torch.float32, 128), (torch.float16, 128),
                                       (torch.float16, 64), (torch.bfloat16, 16)])
def test_forward_mean_segment_edges(dtype, dim):
    batch = 260
    tables, ind, off, w = _problem((dim, dim), dtype, batch, seed=7 * dim)
    m = _tbe(tables, "mean")
    y = m.forward(ind.to(DEV), off.to(DEV))
    torch.cuda.synchronize()
    ref, scale = forward_reference(tables, batch, ind, off, None, True)
    err = np.abs(y.cpu().double().numpy() - ref)
    assert (err <= 1e-6 * scale + 1e-30).all()  # one rounding of a sum that is exact


@pytest.mark.parametrize("dtype,dim", [(torch.float32, 128), (torch.float16, 128),
                                       (torch.float16, 64), (torch.float32, 16)])
def test_forward_out_of_range_lookups_add_nothing(dtype, dim):
    # Scattered bad ids put padding-free batches on the checked path too.
    from paper_2609_30656_gb300.tbe import CB_ERR_INDEX_OOB, TBE
    batch = 260
    tables, ind, off, _ = _problem((dim, dim), dtype, batch, seed=11 * dim, empty_table=False)
    g = torch.Generator().manual_seed(5)
    bad = torch.rand(ind.numel(), generator=g) < 0.01
    rows0 = tables[0].shape[0]
    ind_bad = ind.clone()
    ind_bad[bad] = -3
    m = TBE([t.to(DEV) for t in tables])
    y = m.forward(ind_bad.to(DEV), off.to(DEV))
    torch.cuda.synchronize()
    assert m.get_error() == CB_ERR_INDEX_OOB
    # Reference: the bad lookups read an appended zero row.
    ref_tables = [torch.cat([t, torch.zeros(1, dim, dtype=dtype)]) for t in tables]
    ind_ref = ind.clone()
    t_of = torch.searchsorted(off[::batch][1:], torch.arange(ind.numel()), right=True)
    ind_ref[bad] = torch.tensor([ref_tables[int(t)].shape[0] - 1 for t in t_of[bad]],
                                dtype=torch.int64)
    assert rows0 == ref_tables[0].shape[0] - 1
    ref, _ = forward_reference(ref_tables, batch, ind_ref, off, None, False)
    np.testing.assert_array_equal(y.cpu().double().numpy(), ref)


def _bwd_indices(kind: str, n: int, rows: int, g: torch.Generator) -> torch.Tensor:
    if kind == "distinct":  # every run one long
        return torch.randperm(max(rows, n), generator=g)[:n] % rows
    if kind == "runs32":  # runs exactly one batch long
        return (torch.arange(n) // 32) % rows
    if kind == "hot":  # a few rows repeated thousands of times, the rest rare
        hot = torch.randint(0, 4, (n,), generator=g)
        cold = torch.randint(0, rows, (n,), generator=g)
        return torch.where(torch.rand(n, generator=g) < 0.7, hot, cold)
    raise KeyError(kind)


@pytest.mark.parametrize("dim", BWD_DIMS)
@pytest.mark.parametrize("kind", ["distinct", "runs32", "hot"])
@pytest.mark.parametrize("weighted", [False, True])
def test_backward_run_edges_bit_exact(dim, kind, weighted):
    batch = 260
    tables, ind, off, w = _problem((dim, dim, dim), torch.float32, batch, seed=3 * dim,
                                   weighted=weighted)
    rows, dims = table_meta(tables)
    g = torch.Generator().manual_seed(dim)
    parts = []
    for t in range(3):
        s, e = int(off[t * batch]), int(off[(t + 1) * batch])
        parts.append(_bwd_indices(kind, e - s, int(rows[t]), g))
    ind = torch.cat(parts)
    go = torch.randint(-8, 9, (batch, int(dims.sum())), generator=g).to(torch.float32)
    m = _tbe(tables)
    gr = m.backward(ind.to(DEV), off.to(DEV), go.to(DEV), None if w is None else w.to(DEV))
    torch.cuda.synchronize()
    res, _ = backward_reference(rows, dims, batch, ind, off, go, w, False)
    U = gr.num_unique
    assert U == res.num_unique
    np.testing.assert_array_equal(gr.unique_ids[:U].cpu().numpy(), res.uniq)
    np.testing.assert_array_equal(gr.grad_offsets[:U + 1].cpu().numpy(), res.grad_offsets)
    np.testing.assert_array_equal(gr.table_offsets.cpu().numpy(), res.table_offsets)
    np.testing.assert_array_equal(gr.grads[:gr.num_floats].cpu().double().numpy(), res.grads)
