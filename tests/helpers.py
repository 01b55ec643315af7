"""Shared test helpers: small random problems and torch-CPU float64 cross-checks.

The torch routines here are an independent library statement of the same
quantities (torch.nn.functional.embedding_bag and its autograd), used only to
pin the oracle; the CUDA path is never compared against them.
"""

from __future__ import annotations

import numpy as np
import torch
import torch.nn.functional as F

from paper_2609_30656_gb300 import workloads as wl


def random_problem(seed: int, dims=(8, 16, 24), rows=(7, 50, 13), batch=9, max_len=12,
                   dtype=torch.float32, int_valued=False, weighted=False, empty_frac=0.2):
    """Tables, key-major offsets and indices with ragged (and empty) bags."""
    g = torch.Generator().manual_seed(seed)
    tables = []
    for r, d in zip(rows, dims):
        if int_valued:
            x = torch.randint(-8, 9, (r, d), generator=g).to(torch.float32)
        else:
            x = torch.randn(r, d, generator=g)
        tables.append(x.to(dtype))
    lens = torch.randint(0, max_len + 1, (len(rows) * batch,), generator=g)
    lens[torch.rand(lens.shape, generator=g) < empty_frac] = 0
    offsets = torch.zeros(lens.numel() + 1, dtype=torch.int64)
    offsets[1:] = torch.cumsum(lens, 0)
    idx = []
    for t, r in enumerate(rows):
        s, e = int(offsets[t * batch]), int(offsets[(t + 1) * batch])
        idx.append(torch.randint(0, r, (e - s,), generator=g))
    indices = torch.cat(idx) if idx else torch.zeros(0, dtype=torch.int64)
    weights = None
    if weighted:
        if int_valued:
            weights = torch.randint(0, 3, (indices.numel(),), generator=g).to(torch.float32)
        else:
            weights = torch.rand(indices.numel(), generator=g)
    return tables, indices, offsets, weights


def torch_forward_f64(tables, batch, indices, offsets, weights=None, mean=False):
    """Per-table torch embedding_bag in float64 (include_last_offset)."""
    outs = []
    for t, E in enumerate(tables):
        s, e = int(offsets[t * batch]), int(offsets[(t + 1) * batch])
        off_t = (offsets[t * batch:(t + 1) * batch + 1] - s).to(torch.int64)
        ind_t = indices[s:e].to(torch.int64)
        W = E.to(torch.float64)
        if weights is None:
            y = F.embedding_bag(ind_t, W, off_t, mode="mean" if mean else "sum",
                                include_last_offset=True)
        else:
            y = F.embedding_bag(ind_t, W, off_t, mode="sum", include_last_offset=True,
                                per_sample_weights=weights[s:e].to(torch.float64))
            if mean:
                L = (off_t[1:] - off_t[:-1]).to(torch.float64)
                y = torch.where(L[:, None] > 0, y / L.clamp(min=1)[:, None], torch.zeros_like(y))
        outs.append(y)
    return torch.cat(outs, dim=1)


def torch_dense_grad_f64(tables, batch, indices, offsets, grad_out, weights=None, mean=False):
    """Dense dE_t from torch autograd through embedding_bag in float64."""
    leaves = [E.to(torch.float64).clone().requires_grad_(True) for E in tables]
    y = torch_forward_f64(leaves, batch, indices, offsets, weights, mean)
    (y * grad_out.to(torch.float64)).sum().backward()
    return [L.grad.detach().clone() for L in leaves]


def sparse_to_dense(res, rows, dims):
    """Scatter an oracle/GPU row-sparse gradient into dense per-table arrays."""
    row_base = np.concatenate([[0], np.cumsum(rows)])
    dense = [np.zeros((int(r), int(d))) for r, d in zip(rows, dims)]
    for u, key in enumerate(np.asarray(res.uniq)):
        t = int(np.searchsorted(row_base, key, side="right") - 1)
        r = int(key - row_base[t])
        go = int(res.grad_offsets[u])
        dense[t][r] = res.grads[go:go + dims[t]]
    return dense


def table_meta(tables):
    return (np.array([E.shape[0] for E in tables], dtype=np.int64),
            np.array([E.shape[1] for E in tables], dtype=np.int32))


__all__ = ["random_problem", "torch_forward_f64", "torch_dense_grad_f64", "sparse_to_dense",
           "table_meta", "wl"]


# ----------------------------------------------------------------------------- GPU parity

RTOL = {torch.float32: 1e-5, torch.float16: 2e-3, torch.bfloat16: 2e-3}
RTOL_BWD = 1e-5  # gradients are accumulated and stored in fp32 whatever the table dtype


def forward_reference(tables_cpu, batch, indices, offsets, weights, mean):
    """Oracle output and its condition scale S = s_b * sum_i |w_i * E[idx_i, j]|."""
    import oracle
    ref = oracle.forward(tables_cpu, batch, indices, offsets, weights=weights, mean=mean)
    absw = None if weights is None else weights.abs()
    scale = oracle.forward([t.abs() for t in tables_cpu], batch, indices, offsets, weights=absw,
                           mean=mean)
    return ref, scale


def assert_forward_close(y_gpu, ref, scale, rtol, what=""):
    y = y_gpu.detach().cpu().double().numpy()
    assert y.shape == ref.shape
    err = np.abs(y - ref)
    bad = err > rtol * scale + 1e-30
    if bad.any():
        i = np.argwhere(bad)[0]
        raise AssertionError(f"{what}: {int(bad.sum())} elements off; first at {tuple(i)}: "
                             f"gpu {y[tuple(i)]!r} oracle {ref[tuple(i)]!r} scale {scale[tuple(i)]!r}")


def backward_reference(rows, dims, batch, indices, offsets, grad_out, weights, mean):
    import oracle
    res = oracle.backward(rows, dims, batch, indices, offsets, grad_out, weights=weights, mean=mean)
    absw = None if weights is None else weights.abs()
    sc = oracle.backward(rows, dims, batch, indices, offsets, grad_out.abs(), weights=absw,
                         mean=mean)
    return res, sc.grads


def assert_backward_matches(g, res, scale, rtol=RTOL_BWD, what=""):
    U = g.num_unique
    assert U == res.num_unique, f"{what}: U {U} vs oracle {res.num_unique}"
    F = g.num_floats
    assert F == int(res.grad_offsets[-1])
    np.testing.assert_array_equal(g.unique_ids[:U].cpu().numpy(), res.uniq)
    np.testing.assert_array_equal(g.table_offsets.cpu().numpy(), res.table_offsets)
    np.testing.assert_array_equal(g.grad_offsets[:U + 1].cpu().numpy(), res.grad_offsets)
    got = g.grads[:F].detach().cpu().double().numpy()
    err = np.abs(got - res.grads)
    bad = err > rtol * scale + 1e-30
    if bad.any():
        i = int(np.argwhere(bad)[0][0])
        raise AssertionError(f"{what}: {int(bad.sum())} gradient values off; first at {i}: "
                             f"gpu {got[i]!r} oracle {res.grads[i]!r} scale {scale[i]!r}")


def sub_batch(indices, offsets, weights, num_tables, batch, cols):
    """The bags (t, b) for b in `cols` of every table, as a smaller key-major batch."""
    cols = torch.as_tensor(cols, dtype=torch.int64)
    off = offsets.cpu()
    ind = indices.cpu()
    w = None if weights is None else weights.cpu()
    new_ind, new_w, lens = [], [], []
    for t in range(num_tables):
        for b in cols.tolist():
            s, e = int(off[t * batch + b]), int(off[t * batch + b + 1])
            new_ind.append(ind[s:e])
            if w is not None:
                new_w.append(w[s:e])
            lens.append(e - s)
    o = torch.zeros(len(lens) + 1, dtype=torch.int64)
    o[1:] = torch.cumsum(torch.tensor(lens, dtype=torch.int64), 0)
    ii = torch.cat(new_ind) if new_ind else torch.zeros(0, dtype=ind.dtype)
    ww = (torch.cat(new_w) if new_w else torch.zeros(0)) if w is not None else None
    return ii.to(ind.dtype), o.to(ind.dtype), ww


def compact_tables(tables, indices, offsets, num_tables, batch):
    """Host copies of only the rows a batch touches, with indices renumbered.

    Returns (host tables, renumbered host indices). The renumbering is a plain
    torch.unique / searchsorted per table, so the oracle sees the same stored
    rows at new positions: a pooled sum does not depend on where a row lives.
    """
    off = offsets.cpu()
    new_tabs, new_ind = [], []
    for t in range(num_tables):
        s, e = int(off[t * batch]), int(off[(t + 1) * batch])
        idx = indices[s:e]
        if idx.numel() == 0:
            new_tabs.append(tables[t][:1].cpu())
            new_ind.append(idx.cpu())
            continue
        uniq = torch.unique(idx)
        new_tabs.append(tables[t].index_select(0, uniq.to(tables[t].device)).cpu())
        new_ind.append(torch.searchsorted(uniq, idx).cpu())
    return new_tabs, torch.cat(new_ind).to(indices.dtype) if new_ind else indices.cpu()


def storage_ulp(x: np.ndarray, dtype) -> np.ndarray:
    """Spacing of the storage type at |x| (for a one-rounding allowance)."""
    mant = {torch.float32: 23, torch.float16: 10, torch.bfloat16: 7}[dtype]
    emin = {torch.float32: -126, torch.float16: -14, torch.bfloat16: -126}[dtype]
    e = np.floor(np.log2(np.maximum(np.abs(x), 2.0 ** emin)))
    return 2.0 ** (e - mant)


def bag_of_positions(offsets) -> torch.Tensor:
    """Bag t*B + b of every lookup position (int64 [n]), from key-major offsets."""
    off = torch.as_tensor(offsets).cpu().to(torch.int64)
    lens = off[1:] - off[:-1]
    return torch.repeat_interleave(torch.arange(lens.numel(), dtype=torch.int64), lens)


def inject_out_of_range(tables, indices, offsets, batch, seed, frac=0.05):
    """A copy of `indices` where about `frac` of the lookups of every table hold
    -1 or rows_t instead; returns (indices, bool mask of the replaced lookups)."""
    g = torch.Generator().manual_seed(seed)
    ind = indices.cpu().clone()
    off = offsets.cpu().to(torch.int64)
    bad = torch.rand(ind.numel(), generator=g) < frac
    for t, E in enumerate(tables):
        s, e = int(off[t * batch]), int(off[(t + 1) * batch])
        sel = bad[s:e]
        k = int(sel.sum())
        if k == 0:
            continue
        hi = torch.randint(0, 2, (k,), generator=g).bool()
        vals = torch.where(hi, torch.full((k,), int(E.shape[0])), torch.full((k,), -1))
        part = ind[s:e]
        part[sel] = vals.to(ind.dtype)
    return ind, bad


def without_lookups(indices, offsets, weights, drop, mean):
    """The batch with the lookups where `drop` is set removed, as the library
    treats them: they add nothing, and for mean pooling the bag length still
    counts them. A mean-pooled batch therefore becomes a sum-pooled one whose
    weights are w_i / L (L the original length, rounded to fp32 as the library
    rounds its coefficient). Returns (indices, offsets, weights or None)."""
    off = torch.as_tensor(offsets).cpu().to(torch.int64)
    ind = torch.as_tensor(indices).cpu()
    bag = bag_of_positions(off)
    keep = ~drop
    lens = off[1:] - off[:-1]
    kept = torch.bincount(bag[keep], minlength=lens.numel())
    new_off = torch.zeros(lens.numel() + 1, dtype=torch.int64)
    new_off[1:] = torch.cumsum(kept, 0)
    w = None if weights is None else torch.as_tensor(weights).cpu().to(torch.float32)
    if mean:
        base = torch.ones(ind.numel(), dtype=torch.float32) if w is None else w
        w = base / lens[bag].to(torch.float32)
    return (ind[keep].contiguous(), new_off.to(ind.dtype),
            None if w is None else w[keep].contiguous())
